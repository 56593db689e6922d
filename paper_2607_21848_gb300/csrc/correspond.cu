// Depth-reprojection correspondence (Sec. 4.3, Eq. 3) with the occlusion-aware
// visibility test (Eq. 4) and the exact-fallback rules of the design choices.
//
// Pairs (query token p, source frame s) are laid out [N_q][S].  Per (target frame
// t, source frame s) the kernel composes, at block start,
//     M_ts = K_s R_s^T R_t K_t^-1,   m_ts = K_s R_s^T (c_t - c_s),
// so that for a query at grid cell (j, i) with depth z
//     K_s X_s = z M_ts (j, i, 1)^T + m_ts        (X_s of Eq. 3),
// whose last component is [X_s]_z (K_s's last row is (0, 0, 1)), and
//     u^ = pi(K_s X_s) = (first two components) / [X_s]_z.
// The composition runs in fp32 -- the per-pair arithmetic that consumes it is fp32
// anyway -- except for the camera-centre difference, formed in fp64 so that nearby
// centres do not cancel.  The frame records are stored as fp64; their conversion to
// fp32 runs on the integer pipe, since this GPU's fp64 and conversion throughput is
// a small fraction of its fp32 and integer throughput and every block repeats it.
//
// The launch allows programmatic stream serialization: a block first does the work
// that depends on its arguments alone, then waits for the grid before it
// (griddepcontrol.wait) before it reads bank data or depths or writes an output, and
// it lets the next grid begin its launch as soon as it starts, so that launch latency
// overlaps the running grid.  Depths are read through the read-only data path; the
// outputs, written once and read by a later kernel, are stored streaming (evict first),
// which took the 126 MB sweep from 27.1-27.3 to 24.2-24.4 us.
#include <math.h>

#include "internal.cuh"

namespace crc {

namespace {

constexpr int kMaxS = CRC_MAX_K * CRC_MAX_FRAMES;
constexpr int kMaxPairs = CRC_MAX_FRAMES * kMaxS;
// frame values loaded per prologue thread: 4 (256 - 31 - 32) >= 21 kMaxS
constexpr int kLoadsPerThread = 4;
static_assert(kLoadsPerThread * (256 - 31 - 32) >= kFrameDoubles * kMaxS, "prologue loads do not cover the records");

// 16 words, 16-byte aligned
struct __align__(16) PairXf {
  float M[9];     // M_ts = K_s A_ts, A_ts = R_s^T R_t K_t^-1; its last row is A_ts's
  float m[3];     // m_ts = K_s b_ts, b_ts = R_s^T (c_t - c_s); NaN when the pair is not a retrieval, so that u^ is NaN
  int depth_off;  // offset of D_s in the bank depth array, -1 if the pair is not a retrieval
  int pad[3];
};

// IEEE-754 binary64 -> binary32, round to nearest even, on the integer pipe (this
// GPU's fp64 and conversion rates are a small fraction of its integer rate).
// Results below the binary32 normal range become signed zero.
__device__ __forceinline__ float f64_to_f32(double x) {
  const unsigned long long u = (unsigned long long)__double_as_longlong(x);
  const unsigned sign = (unsigned)(u >> 32) & 0x80000000u;
  const int e = (int)((u >> 52) & 0x7ff) - 1023 + 127;
  if (e <= 0) return __uint_as_float(sign);
  if (e >= 255) return __uint_as_float(sign | 0x7f800000u);
  const unsigned long long mant = u & 0xfffffffffffffull;
  unsigned r = ((unsigned)e << 23) | (unsigned)(mant >> 29);
  const unsigned rest = (unsigned)(mant & 0x1fffffffull);
  if (rest > 0x10000000u || (rest == 0x10000000u && (r & 1u))) ++r;  // a carry moves into the exponent
  return __uint_as_float(sign | r);
}

// packed fp32 pairs (f32x2 ALU ops): each lane rounds exactly as the scalar op does
__device__ __forceinline__ uint64_t pk2(float a, float b) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ void upk2(uint64_t r, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(r));
}
__device__ __forceinline__ uint64_t ffma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t fmul2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

__device__ void mat3_inverse(const float* m, float* inv) {
  const float c00 = m[4] * m[8] - m[5] * m[7];
  const float c01 = m[5] * m[6] - m[3] * m[8];
  const float c02 = m[3] * m[7] - m[4] * m[6];
  const float det = m[0] * c00 + m[1] * c01 + m[2] * c02;
  const float id = 1.0f / det;
  inv[0] = c00 * id;
  inv[1] = (m[2] * m[7] - m[1] * m[8]) * id;
  inv[2] = (m[1] * m[5] - m[2] * m[4]) * id;
  inv[3] = c01 * id;
  inv[4] = (m[0] * m[8] - m[2] * m[6]) * id;
  inv[5] = (m[2] * m[3] - m[0] * m[5]) * id;
  inv[6] = c02 * id;
  inv[7] = (m[1] * m[6] - m[0] * m[7]) * id;
  inv[8] = (m[0] * m[4] - m[1] * m[3]) * id;
}

}  // namespace

// VIS: the visibility test of Eq. 4 is in force (eps finite).  P: source frames per
// thread (2 when S is even and the outputs are aligned for 16-byte stores).
template <int P, bool VIS, typename Idx>
__global__ void __launch_bounds__(256, 4) correspond_kernel(const __grid_constant__ CorrespondArgs a, int FL) {
  __shared__ PairXf px[kMaxPairs];
  __shared__ float src_KR[kMaxS][18];   // K_s, R_s
  __shared__ double src_c[kMaxS][3];    // c_s
  __shared__ int src_off[kMaxS];
  __shared__ float tgt_RK[CRC_MAX_FRAMES][9];  // R_t K_t^-1
  __shared__ double tgt_c[CRC_MAX_FRAMES][3];  // c_t
  // the next grid may begin its launch at once: this grid is one wave, so nothing of it
  // waits for SM space, and the next grid's blocks wait for this one before they read
  asm volatile("griddepcontrol.launch_dependents;");
  const int S = a.k * a.F;
  const int hw = a.h * a.w;
  const int Nq = a.F * hw;
  const int L = S / P;           // threads per query
  const int R = blockDim.x / L;  // queries per block step
  const int steps = ((Nq + R - 1) / R + gridDim.x - 1) / gridDim.x;
  const int qb = blockIdx.x * steps * R;
  const int q_end = min(Nq, qb + steps * R);
  if (qb >= q_end) return;  // the whole block
  const int t_lo = qb / hw, nt = (q_end - 1) / hw - t_lo + 1;
  // Thread (g, qi, fi) handles source frames s0 = g FL + P fi .. s0 + P - 1 of
  // queries qb + qi, qb + qi + R, ...: a warp covers 32 P / FL adjacent queries x FL
  // frames, so that its source-depth reads fall into few lines while each query's FL
  // outputs stay contiguous.  A block step writes R S consecutive pairs.
  const int i = threadIdx.x;
  const int FLP = FL / P;
  const int fi = i % FLP;
  const int qi = (i / FLP) % R;
  const int s0 = (i / (FLP * R)) * FL + fi * P;
  int q = qb + qi;

  // Warp 0 forms R_t K_t^-1 for the block's target frames from the kernel arguments
  // alone, before the wait on the grid this launch depends on; everything below reads
  // data that grid may write (indices, bank records, depths) or writes outputs.
  if (i < nt) {
    const int t = t_lo + i;
    const double* ft = a.step ? reinterpret_cast<const double*>(&a.step->frames[t]) : &a.cur.rec[t][0];
    float Kt[9], Rt[9], Ki[9];
    for (int e = 0; e < 9; ++e) {
      Kt[e] = f64_to_f32(ft[e]);
      Rt[e] = f64_to_f32(ft[9 + e]);
    }
    mat3_inverse(Kt, Ki);
    for (int m = 0; m < 3; ++m)
      for (int n = 0; n < 3; ++n)
        tgt_RK[i][3 * m + n] = Rt[3 * m + 0] * Ki[n] + Rt[3 * m + 1] * Ki[3 + n] + Rt[3 * m + 2] * Ki[6 + n];
    for (int e = 0; e < 3; ++e) tgt_c[i][e] = ft[18 + e];
  }
  asm volatile("griddepcontrol.wait;" ::: "memory");
  float z = q < q_end ? a.depth[q] : 0.f;  // the first query's depth, in flight through the prologue
  // The source values (21 per source frame) are loaded and converted by all threads
  // but the first warp, in two rounds of independent loads: the slot indices, then
  // the records.  A block has at least 256 - 31 threads (a multiple of S / P <= 32),
  // so kLoadsPerThread loads per thread cover the 21 S <= 672 values.
  if (i >= 32) {
    const int nthr = blockDim.x - 32;
    const int nv = S * kFrameDoubles;
    const int cnt = a.d_count ? *a.d_count : CRC_MAX_K;
    int jr[kLoadsPerThread];
#pragma unroll
    for (int u = 0; u < kLoadsPerThread; ++u) {
      const int v = i - 32 + u * nthr;
      jr[u] = v < nv ? a.d_idx[(v / kFrameDoubles) / a.F] : -1;
    }
    double xv[kLoadsPerThread];
#pragma unroll
    for (int u = 0; u < kLoadsPerThread; ++u) {
      const int v = i - 32 + u * nthr;
      xv[u] = 0.0;
      if (v < nv) {
        const int s = v / kFrameDoubles, e = v - s * kFrameDoubles;
        const int r = s / a.F, f = s - r * a.F;
        const int j = jr[u];
        const bool ok = (j >= 0) && (j < a.capacity) && (r < cnt);
        if (e == 0) src_off[s] = ok ? (int)(((size_t)j * a.F + f) * hw) : -1;
        if (ok) xv[u] = a.bank_frames[((size_t)j * a.F + f) * kFrameDoubles + e];
      }
    }
#pragma unroll
    for (int u = 0; u < kLoadsPerThread; ++u) {
      const int v = i - 32 + u * nthr;
      if (v < nv) {
        const int s = v / kFrameDoubles, e = v - s * kFrameDoubles;
        if (e < 18)
          src_KR[s][e] = f64_to_f32(xv[u]);
        else
          src_c[s][e - 18] = xv[u];
      }
    }
  }
  __syncthreads();
  if (i < nt * S) {
    const int tl = i / S, s = i - (i / S) * S;
    PairXf x;
    x.pad[0] = x.pad[1] = x.pad[2] = 0;
    x.depth_off = src_off[s];
    if (x.depth_off >= 0) {
      const float* Ks = &src_KR[s][0];
      const float* Rs = &src_KR[s][9];
      const float* RK = &tgt_RK[tl][0];
      float A[9], b[3];
      // A = R_s^T (R_t K_t^-1), b = R_s^T (c_t - c_s) with the difference formed in fp64
      for (int m = 0; m < 3; ++m)
        for (int n = 0; n < 3; ++n) A[3 * m + n] = Rs[m] * RK[n] + Rs[3 + m] * RK[3 + n] + Rs[6 + m] * RK[6 + n];
      float dc[3];
      for (int e = 0; e < 3; ++e) dc[e] = f64_to_f32(tgt_c[tl][e] - src_c[s][e]);
      for (int m = 0; m < 3; ++m) b[m] = Rs[m] * dc[0] + Rs[3 + m] * dc[1] + Rs[6 + m] * dc[2];
      // M = K_s A and m = K_s b; the last rows are A's and b's
      for (int m = 0; m < 2; ++m) {
        for (int n = 0; n < 3; ++n) x.M[3 * m + n] = Ks[3 * m] * A[n] + Ks[3 * m + 1] * A[3 + n] + Ks[3 * m + 2] * A[6 + n];
        x.m[m] = Ks[3 * m] * b[0] + Ks[3 * m + 1] * b[1] + Ks[3 * m + 2] * b[2];
      }
      for (int n = 0; n < 3; ++n) x.M[6 + n] = A[6 + n];
      x.m[2] = b[2];
    } else {
      for (int e = 0; e < 9; ++e) x.M[e] = 0.f;
      x.m[0] = x.m[1] = x.m[2] = __int_as_float(0x7fc00000);
    }
    px[i] = x;
  }
  __syncthreads();

  if (q >= q_end) return;
  int t = q / hw;
  int iy = (q - t * hw) / a.w;
  int jx = q - t * hw - iy * a.w;
  // the (t, s) transforms of the thread's P frames, lane p of each packed pair for s0 + p
  float c0[P], c1[P], c2[P], r0[P], r1[P], r2[P], m0[P], m1[P], m2[P];
  int doff[P];
#pragma unroll
  for (int p = 0; p < P; ++p) {
    const PairXf& x = px[(t - t_lo) * S + s0 + p];
    c0[p] = x.M[0], c1[p] = x.M[3], c2[p] = x.M[6];
    r0[p] = fmaf(x.M[1], (float)iy, x.M[2]);
    r1[p] = fmaf(x.M[4], (float)iy, x.M[5]);
    r2[p] = fmaf(x.M[7], (float)iy, x.M[8]);
    m0[p] = x.m[0], m1[p] = x.m[1], m2[p] = x.m[2];
    doff[p] = x.depth_off;
  }
  const float one_eps = 1.0f + a.eps;
  const float wf = (float)a.w, hf = (float)a.h;
  Idx o = (Idx)q * (Idx)S + (Idx)s0;
  const Idx o_step = (Idx)R * (Idx)S;
  for (; q < q_end; q += R, o += o_step) {
    const float zn = q + R < q_end ? __ldg(a.depth + q + R) : 0.f;  // next query's depth, in flight meanwhile
    const float u0 = (float)jx;
    const bool z_ok = (z > 0.f) & (z < INFINITY);
    float ux[P], uy[P], X2[P];
    if (P == 2) {
      // K_s X_s = z M (j, i, 1)^T + m for both frames at once; its last component is [X_s]_z
      const uint64_t U0 = pk2(u0, u0), Z = pk2(z, z);
      const uint64_t X0 = ffma2(Z, ffma2(pk2(c0[0], c0[P - 1]), U0, pk2(r0[0], r0[P - 1])), pk2(m0[0], m0[P - 1]));
      const uint64_t X1 = ffma2(Z, ffma2(pk2(c1[0], c1[P - 1]), U0, pk2(r1[0], r1[P - 1])), pk2(m1[0], m1[P - 1]));
      const uint64_t XZ = ffma2(Z, ffma2(pk2(c2[0], c2[P - 1]), U0, pk2(r2[0], r2[P - 1])), pk2(m2[0], m2[P - 1]));
      upk2(XZ, X2[0], X2[P - 1]);
      float iq0, iq1;
      asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(iq0) : "f"(X2[0]));
      asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(iq1) : "f"(X2[P - 1]));
      const uint64_t IQ = pk2(iq0, iq1);
      upk2(fmul2(X0, IQ), ux[0], ux[P - 1]);
      upk2(fmul2(X1, IQ), uy[0], uy[P - 1]);
    } else {
      const float X0 = fmaf(z, fmaf(c0[0], u0, r0[0]), m0[0]);
      const float X1 = fmaf(z, fmaf(c1[0], u0, r1[0]), m1[0]);
      X2[0] = fmaf(z, fmaf(c2[0], u0, r2[0]), m2[0]);
      float iq;
      asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(iq) : "f"(X2[0]));  // 1 ulp; a subnormal X2 gives inf, hence invalid
      ux[0] = X0 * iq;
      uy[0] = X1 * iq;
    }
    bool ok[P];
    int cell[P];
#pragma unroll
    for (int p = 0; p < P; ++p) {
      const float vx = ux[p] + 0.5f, vy = uy[p] + 0.5f;
      // the nearest cell is floor(u^ + 1/2); every comparison fails on NaN
      ok[p] = z_ok & (X2[p] > 0.f) & (X2[p] < INFINITY) & (vx >= 0.f) & (vx < wf) & (vy >= 0.f) & (vy < hf);
      cell[p] = ok[p] ? __float2int_rd(vy) * a.w + __float2int_rd(vx) : -1;
    }
    if (VIS) {
      float ds[P];
#pragma unroll
      for (int p = 0; p < P; ++p) ds[p] = __ldg(ok[p] ? a.bank_depth + (doff[p] + cell[p]) : a.depth + q);
#pragma unroll
      for (int p = 0; p < P; ++p) {
        ok[p] = ok[p] & (X2[p] <= one_eps * ds[p]);
        cell[p] = ok[p] ? cell[p] : -1;
      }
    }
    if (P == 2) {
      __stcs(reinterpret_cast<float4*>(a.uv + 2 * o), make_float4(ux[0], uy[0], ux[P - 1], uy[P - 1]));
      if (a.cell) __stcs(reinterpret_cast<int2*>(a.cell + o), make_int2(cell[0], cell[P - 1]));
      __stcs(reinterpret_cast<unsigned short*>(a.valid + o), (unsigned short)((ok[0] ? 1u : 0u) | (ok[P - 1] ? 0x100u : 0u)));
    } else {
      __stcs(reinterpret_cast<float2*>(a.uv) + o, make_float2(ux[0], uy[0]));
      if (a.cell) __stcs(a.cell + o, cell[0]);
      __stcs(reinterpret_cast<unsigned char*>(a.valid) + o, (unsigned char)(ok[0] ? 1 : 0));
    }
    jx += R;
    if (jx >= a.w) {
      const int t_was = t;
      do {
        jx -= a.w;
        if (++iy == a.h) {
          iy = 0;
          ++t;
        }
      } while (jx >= a.w);
      if (t < a.F) {
#pragma unroll
        for (int p = 0; p < P; ++p) {
          const PairXf& x = px[(t - t_lo) * S + s0 + p];
          if (t != t_was) {
            c0[p] = x.M[0], c1[p] = x.M[3], c2[p] = x.M[6];
            m0[p] = x.m[0], m1[p] = x.m[1], m2[p] = x.m[2];
            doff[p] = x.depth_off;
          }
          r0[p] = fmaf(x.M[1], (float)iy, x.M[2]);
          r1[p] = fmaf(x.M[4], (float)iy, x.M[5]);
          r2[p] = fmaf(x.M[7], (float)iy, x.M[8]);
        }
      }
    }
    z = zn;
  }
}

template <int P, bool VIS, typename Idx>
static cudaError_t launch_v(const CorrespondArgs& a, cudaStream_t s, int sms, int S, int Nq) {
  const int L = S / P;
  const int threads = (256 / L) * L;
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, correspond_kernel<P, VIS, Idx>, threads, 0) !=
          cudaSuccess ||
      per_sm < 1)
    per_sm = 1;
  const int R = threads / L;
  const int groups = (Nq + R - 1) / R;
  const int blocks = groups < per_sm * sms ? groups : per_sm * sms;
  int fl = 8;
  while (S % fl != 0 || fl % P != 0) --fl;  // frames per lane group: the largest divisor of S up to 8 (a multiple of P)
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(blocks);
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, correspond_kernel<P, VIS, Idx>, a, fl);
}

template <int P, typename Idx>
static cudaError_t launch_pi(const CorrespondArgs& a, cudaStream_t s, int sms, int S, int Nq) {
  return isinf(a.eps) ? launch_v<P, false, Idx>(a, s, sms, S, Nq) : launch_v<P, true, Idx>(a, s, sms, S, Nq);
}

cudaError_t launch_correspond(const CorrespondArgs& a, cudaStream_t s) {
  const int Nq = a.F * a.h * a.w;
  const int S = a.k * a.F;
  if (Nq == 0 || S == 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  // two source frames per thread when S is even and the outputs take 16-, 8- and 2-byte stores
  const bool two = S % 2 == 0 && ((uintptr_t)a.uv & 15) == 0 && ((uintptr_t)a.cell & 7) == 0 &&
                   ((uintptr_t)a.valid & 1) == 0;
  const bool narrow = (uint64_t)Nq * (uint64_t)S < (1ull << 32);  // pair offsets fit 32 bits
  if (two)
    return narrow ? launch_pi<2, uint32_t>(a, s, sms, S, Nq) : launch_pi<2, size_t>(a, s, sms, S, Nq);
  return narrow ? launch_pi<1, uint32_t>(a, s, sms, S, Nq) : launch_pi<1, size_t>(a, s, sms, S, Nq);
}

}  // namespace crc
