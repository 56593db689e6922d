// Gather of retrieved chunks from the slab pool into a cache (Sec. 4.2), with the
// optional temporal RoPE re-positioning of the keys (Sec. 4.2 "Cache packing").
//
// Shared by the fused retrieval launch and the standalone mirror gather, so both
// produce bit-identical cache contents for the same slots.
#pragma once

#include <cuda_bf16.h>
#include <stdint.h>

#include "copy.cuh"
#include "internal.cuh"

namespace crc {

// Per-CTA plan of one gather: the chunk held by every slot, whether its keys are
// rotated, and the (cos, sin) of each slot's rotation for every temporal pair.
struct GatherPlan {
  int32_t chunk[CRC_MAX_K];
  int32_t rotate[CRC_MAX_K];
  float2 cs[CRC_MAX_K][CRC_MAX_ROPE_PAIRS];
};

// Position shift of slot r holding chunk j: from frame_pos0 + j*F to pos_slot0 + r*pos_stride.
__device__ __forceinline__ int64_t rope_delta(const GatherArgs& g, int32_t pos_slot0, int r, int64_t j) {
  return (int64_t)pos_slot0 + (int64_t)r * g.rope_pos_stride - ((int64_t)g.rope_frame_pos0 + j * g.F);
}

// Fills plan.rotate[] and plan.cs[] once plan.chunk[] is visible to the whole block.
// Angles are formed in fp64 (delta * omega_i) so that large position shifts keep
// their accuracy; the rotation itself runs in fp32.  Ends with a block barrier.
__device__ inline void plan_rope(const GatherArgs& g, int k, GatherPlan& p, int32_t pos_slot0) {
  for (int r = threadIdx.x; r < k; r += blockDim.x) {
    const int64_t j = p.chunk[r];
    p.rotate[r] = (g.rope_pairs > 0 && j >= 0 && rope_delta(g, pos_slot0, r, j) != 0) ? 1 : 0;
  }
  const int n = k * g.rope_pairs;
  for (int e = threadIdx.x; e < n; e += blockDim.x) {
    const int r = e / g.rope_pairs, i = e - r * g.rope_pairs;
    const int64_t j = p.chunk[r];
    if (j < 0) continue;
    double sn, cn;
    sincos((double)rope_delta(g, pos_slot0, r, j) * g.rope_omega[i], &sn, &cn);
    p.cs[r][i] = make_float2((float)cn, (float)sn);
  }
  __syncthreads();
}

// (a + i b) * (cos + i sin), each product rounded separately.
__device__ __forceinline__ void rotate_pair(float& a, float& b, float2 cs) {
  const float na = __fsub_rn(__fmul_rn(a, cs.x), __fmul_rn(b, cs.y));
  const float nb = __fadd_rn(__fmul_rn(a, cs.y), __fmul_rn(b, cs.x));
  a = na;
  b = nb;
}

// 16-byte vectors of the cache dtype widened to fp32 and rounded back (nearest even).
template <bool BF16>
struct Vec16;

template <>
struct Vec16<true> {
  static constexpr int N = 8;
  __device__ static __forceinline__ void unpack(const uint4& v, float x[8]) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      x[2 * i] = __uint_as_float(w[i] << 16);
      x[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
  }
  __device__ static __forceinline__ uint4 pack(const float x[8]) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const __nv_bfloat162 h = __floats2bfloat162_rn(x[2 * i], x[2 * i + 1]);
      w[i] = *reinterpret_cast<const uint32_t*>(&h);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
  }
};

template <>
struct Vec16<false> {
  static constexpr int N = 4;
  __device__ static __forceinline__ void unpack(const uint4& v, float x[4]) {
    x[0] = __uint_as_float(v.x);
    x[1] = __uint_as_float(v.y);
    x[2] = __uint_as_float(v.z);
    x[3] = __uint_as_float(v.w);
  }
  __device__ static __forceinline__ uint4 pack(const float x[4]) {
    return make_uint4(__float_as_uint(x[0]), __float_as_uint(x[1]), __float_as_uint(x[2]), __float_as_uint(x[3]));
  }
};

// One 16-byte vector of interleaved pairs: the pairs whose bit is set in `rot` are
// rotated by f[] (as rotate_pair, rounded back to the cache dtype); the others keep
// their bits exactly.  Every lane runs the same instructions, whatever its pairs.
template <bool BF16>
__device__ __forceinline__ uint4 rotate_interleaved(const uint4& v, const float2* f, uint32_t rot) {
  uint32_t w[4] = {v.x, v.y, v.z, v.w};
  if constexpr (BF16) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {  // word i holds pair i
      float a = __uint_as_float(w[i] << 16), b = __uint_as_float(w[i] & 0xffff0000u);
      rotate_pair(a, b, f[i]);
      const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
      const uint32_t nw = *reinterpret_cast<const uint32_t*>(&h);
      w[i] = ((rot >> i) & 1u) ? nw : w[i];
    }
  } else {
#pragma unroll
    for (int i = 0; i < 2; ++i) {  // words 2i, 2i + 1 hold pair i
      float a = __uint_as_float(w[2 * i]), b = __uint_as_float(w[2 * i + 1]);
      rotate_pair(a, b, f[i]);
      const bool on = ((rot >> i) & 1u) != 0;
      w[2 * i] = on ? __float_as_uint(a) : w[2 * i];
      w[2 * i + 1] = on ? __float_as_uint(b) : w[2 * i + 1];
    }
  }
  return make_uint4(w[0], w[1], w[2], w[3]);
}

// One key row (H heads of d channels) copied by a warp with the temporal pairs of
// every head rotated by cs[i].  Interleaved pairs lie inside one 16-byte vector
// (channel0 is even).  Half-split pairs (c, c + pairs) lie in two vectors `half`
// apart (channel0 and pairs are multiples of the vector width); the lane that
// owns the lower vector rotates and writes both.  A lane keeps one vector (two for
// a half-split pair) in flight: that holds the kernel to 61 registers, so that four
// blocks share an SM as in the plain copy, which measured 5220 GB/s on a 30-layer
// re-positioning gather against 4310 with two vectors in flight at 93 registers.
//
// When the vectors of a head divide the warp (d / N in {1, 2, 4, 8, 16, 32}), lane l
// meets the same channels (l mod d/N) * N in every head it copies, so its kind of
// vector and its (cos, sin) factors are fixed for the whole row: taken once, in
// registers.  Other head sizes take the general per-vector path.
template <bool BF16>
__device__ void copy_row_rotated(const char* __restrict__ src, char* __restrict__ dst, const GatherArgs& g,
                                 const float2* __restrict__ cs, int lane) {
  using IO = Vec16<BF16>;
  constexpr int N = IO::N;
  const uint4* s = reinterpret_cast<const uint4*>(src);
  uint4* d = reinterpret_cast<uint4*>(dst);
  const int n = g.row_bytes >> 4;
  const int vph = g.d / N;  // vectors per head
  const int c0 = g.rope_c0, np = g.rope_pairs, np2 = 2 * g.rope_pairs;
  const int half = np / N;
  if ((32 % vph) == 0 && g.rope_interleaved) {
    // interleaved pairs, lane l meeting the same channels in every head: the row is
    // copied like a plain row (four vectors in flight per lane, L2-only loads,
    // streaming stores), each vector passed through the lane's fixed rotation (a
    // no-op select on lanes without rotated pairs)
    const int ch = (lane % vph) * N;
    constexpr int NP = N / 2;
    uint32_t rot = 0u;
    float2 f[NP];
#pragma unroll
    for (int i = 0; i < NP; ++i) {
      const int che = ch + 2 * i;
      const bool in = che >= c0 && che < c0 + np2;
      rot |= in ? (1u << i) : 0u;
      f[i] = in ? cs[(che - c0) >> 1] : make_float2(1.f, 0.f);
    }
    int c = lane;
    for (; c + 96 < n; c += 128) {
      const uint4 a0 = __ldcg(s + c), a1 = __ldcg(s + c + 32), a2 = __ldcg(s + c + 64), a3 = __ldcg(s + c + 96);
      __stcs(d + c, rotate_interleaved<BF16>(a0, f, rot));
      __stcs(d + c + 32, rotate_interleaved<BF16>(a1, f, rot));
      __stcs(d + c + 64, rotate_interleaved<BF16>(a2, f, rot));
      __stcs(d + c + 96, rotate_interleaved<BF16>(a3, f, rot));
    }
    for (; c < n; c += 32) __stcs(d + c, rotate_interleaved<BF16>(__ldcg(s + c), f, rot));
    return;
  }
  if ((32 % vph) == 0) {
    const int ch = (lane % vph) * N;
    const int kind = g.rope_interleaved ? ((ch + N > c0 && ch < c0 + np2) ? 1 : 0)
                                        : ((ch >= c0 && ch < c0 + np) ? 2 : ((ch >= c0 + np && ch < c0 + np2) ? 3 : 0));
    if (kind == 3) return;  // the lane owning the lower half writes this vector
    float2 f[N];            // (cos, sin) of each element's pair; (1, 0) outside the block
#pragma unroll
    for (int e = 0; e < N; ++e) {
      const int i = kind == 1 ? (ch + e - c0) >> 1 : ch - c0 + e;
      const bool in = kind == 1 ? (ch + e >= c0 && ch + e < c0 + np2) : (kind == 2);
      f[e] = in ? cs[i] : make_float2(1.f, 0.f);
    }
    for (int c = lane; c < n; c += 32) {
      const uint4 v = __ldcg(s + c);
      if (kind == 0) {
        d[c] = v;
      } else if (kind == 1) {
        float x[N];
        IO::unpack(v, x);
#pragma unroll
        for (int e = 0; e < N; e += 2) rotate_pair(x[e], x[e + 1], f[e]);
        d[c] = IO::pack(x);
      } else {
        float x[N], y[N];
        IO::unpack(v, x);
        IO::unpack(__ldcg(s + c + half), y);
#pragma unroll
        for (int e = 0; e < N; ++e) rotate_pair(x[e], y[e], f[e]);
        d[c] = IO::pack(x);
        d[c + half] = IO::pack(y);
      }
    }
    return;
  }
  for (int c = lane; c < n; c += 32) {
    const int ch = (c % vph) * N;
    const int kind = g.rope_interleaved
                         ? ((ch + N > c0 && ch < c0 + np2) ? 1 : 0)
                         : ((ch >= c0 && ch < c0 + np) ? 2 : ((ch >= c0 + np && ch < c0 + np2) ? 3 : 0));
    if (kind == 0) {
      d[c] = __ldcg(s + c);
    } else if (kind == 1) {
      float x[N];
      IO::unpack(__ldcg(s + c), x);
#pragma unroll
      for (int e = 0; e < N; e += 2) {
        const int che = ch + e;
        if (che >= c0 && che < c0 + np2) rotate_pair(x[e], x[e + 1], cs[(che - c0) >> 1]);
      }
      d[c] = IO::pack(x);
    } else if (kind == 2) {
      float x[N], y[N];
      IO::unpack(__ldcg(s + c), x);
      IO::unpack(__ldcg(s + c + half), y);
#pragma unroll
      for (int e = 0; e < N; ++e) rotate_pair(x[e], y[e], cs[ch - c0 + e]);
      d[c] = IO::pack(x);
      d[c + half] = IO::pack(y);
    }
  }
}

// Copies every active slot's K and V rows (one warp per token row, rows ordered
// (active slot, K|V, layer, token)) from its slab into the slot's cache segment.
// ROPE = false compiles the plain copy only (no re-positioning requested), which
// keeps the register footprint, and so the copy's occupancy, of a plain gather.
template <bool ROPE>
__device__ inline void gather_slots(const GatherArgs& g, int k, const GatherPlan& p) {
  int act[CRC_MAX_K];
  int n_act = 0;
  for (int r = 0; r < k; ++r)
    if (p.chunk[r] >= 0 && g.slot_offset[r] >= 0) act[n_act++] = r;
  const int64_t rows_per_kv = (int64_t)g.L * g.Nc;
  const int64_t total = (int64_t)n_act * 2 * rows_per_kv;
  const int lane = threadIdx.x & 31;
  const int gwarp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int nwarps = (gridDim.x * blockDim.x) >> 5;
  for (int64_t row = gwarp; row < total; row += nwarps) {
    const int ai = (int)(row / (2 * rows_per_kv));
    int64_t rem = row - (int64_t)ai * 2 * rows_per_kv;
    const int kv = (int)(rem / rows_per_kv);
    rem -= kv * rows_per_kv;
    const int l = (int)(rem / g.Nc);
    const int t = (int)(rem - (int64_t)l * g.Nc);
    const int r = act[ai];
    const int64_t slab = p.chunk[r] % g.num_slabs;
    const char* src = g.pool + slab * g.slab_bytes + kv * g.kv_bytes + rem * g.row_bytes;
    char* dst = (kv ? g.cache_v : g.cache_k) + l * g.cache_layer_stride +
                (int64_t)(g.slot_offset[r] + t) * g.cache_token_stride;
    if (ROPE && kv == 0 && p.rotate[r]) {
      if (g.elem_bytes == 2)
        copy_row_rotated<true>(src, dst, g, p.cs[r], lane);
      else
        copy_row_rotated<false>(src, dst, g, p.cs[r], lane);
    } else {
      warp_copy_row<1>(src, dst, nullptr, g.row_bytes, lane);
    }
  }
}

}  // namespace crc
