// Biased flash attention on the SIMT pipes in fp32 (Sec. 4.3, Eq. 2).
//
// This is the fp32 path (fp32 inputs, fp32 arithmetic throughout), and the
// reference-precision path for bf16 inputs when CRC_ATTN_SIMT is requested.
// One CTA (4 warps) owns 16 query rows of one (layer, head) and streams the
// key/value tiles of 32 keys through shared memory; lane l scores key l of the
// tile for each of its warp's 4 queries, adds lambda*B from the correspondence of
// that query in the key's source frame (Eq. 2, or the opt-in additive Gaussian
// lambda exp(-d^2 / (2 sigma^2))), and the warp keeps an online softmax.
// The bias is formed per (query, key) in registers and never stored.
#include <cuda_bf16.h>
#include <math.h>

#include "internal.cuh"
#include "keys.cuh"

namespace crc {

namespace {

constexpr int kQB = 16;     // query rows per CTA
constexpr int kKT = 32;     // keys per tile
constexpr int kMaxD = 128;

template <typename T>
__device__ __forceinline__ float to_f(T x);
template <>
__device__ __forceinline__ float to_f<float>(float x) { return x; }
template <>
__device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 x) { return __bfloat162float(x); }

template <typename T>
__device__ __forceinline__ T from_f(float x);
template <>
__device__ __forceinline__ float from_f<float>(float x) { return x; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float x) { return __float2bfloat16_rn(x); }

}  // namespace

template <typename T>
__global__ void __launch_bounds__(128) attn_simt_kernel(const __grid_constant__ AttnArgs a) {
  __shared__ float Qs[kQB][kMaxD];
  __shared__ float Ks[kKT][kMaxD + 1];
  __shared__ float Vs[kKT][kMaxD];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int q0 = blockIdx.x * kQB;
  const int head = blockIdx.y, layer = blockIdx.z;
  const int d = a.d;
  const T* Q = static_cast<const T*>(a.q) + layer * a.q_sl + head * a.q_sh;
  const T* Kp = static_cast<const T*>(a.k) + layer * a.k_sl + head * a.k_sh;
  const T* Vp = static_cast<const T*>(a.v) + layer * a.k_sl + head * a.k_sh;

  for (int e = tid; e < kQB * d; e += blockDim.x) {
    const int r = e / d, c = e - (e / d) * d;
    Qs[r][c] = (q0 + r < a.Nq) ? to_f(Q[(int64_t)(q0 + r) * a.q_st + c]) : 0.f;
  }
  const float scale = rsqrtf((float)d);
  const float nb = a.lambda / (2.f * a.sigma * a.sigma);
  const float ng = 1.f / (2.f * a.sigma * a.sigma);
  const int dpl = d / 32;  // output dims per lane
  float m[4], l[4], acc[4][kMaxD / 32];
#pragma unroll
  for (int qi = 0; qi < 4; ++qi) {
    m[qi] = -INFINITY;
    l[qi] = 0.f;
#pragma unroll
    for (int c = 0; c < kMaxD / 32; ++c) acc[qi][c] = 0.f;
  }

  for (int k0 = 0; k0 < a.Nk; k0 += kKT) {
    __syncthreads();
    for (int e = tid; e < kKT * d; e += blockDim.x) {
      const int r = e / d, c = e - (e / d) * d;
      const bool in = k0 + r < a.Nk;
      Ks[r][c] = in ? to_f(Kp[(int64_t)(k0 + r) * a.k_st + c]) : 0.f;
      Vs[r][c] = in ? to_f(Vp[(int64_t)(k0 + r) * a.k_st + c]) : 0.f;
    }
    __syncthreads();
    const KeyInfo ki = key_info_of(a, k0 + lane);
#pragma unroll
    for (int qi = 0; qi < 4; ++qi) {
      const int qr = warp * 4 + qi;
      const int p = q0 + qr;
      float dot = 0.f;
      for (int e = 0; e < d; ++e) dot = fmaf(Qs[qr][e], Ks[lane][e], dot);
      float logit = dot * scale;
      if (ki.src >= 0 && p < a.Nq) {
        const int64_t pi = (int64_t)p * a.S + ki.src;
        if (a.valid[pi]) {
          const float2 u = reinterpret_cast<const float2*>(a.uv)[pi];
          const float dx = ki.x - u.x, dy = ki.y - u.y;
          if (a.bias_form == 1)
            logit += a.lambda * expf(-ng * (dx * dx + dy * dy));  // opt-in additive Gaussian
          else
            logit -= nb * (dx * dx + dy * dy);  // Eq. 2
        }
      }
      if (!ki.active) logit = -INFINITY;
      if (a.frame_causal && ki.frame > p / (a.h * a.w)) logit = -INFINITY;  // a later frame of this chunk
      float tmax = logit;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, o));
      const float mnew = fmaxf(m[qi], tmax);
      if (mnew == -INFINITY) continue;  // nothing active yet for this row (warp-uniform)
      const float corr = expf(m[qi] - mnew);
      const float pr = expf(logit - mnew);
      float psum = pr;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) psum += __shfl_xor_sync(0xffffffffu, psum, o);
      l[qi] = l[qi] * corr + psum;
      m[qi] = mnew;
#pragma unroll
      for (int c = 0; c < kMaxD / 32; ++c) acc[qi][c] *= corr;
      for (int j = 0; j < kKT; ++j) {
        const float pj = __shfl_sync(0xffffffffu, pr, j);
#pragma unroll
        for (int c = 0; c < kMaxD / 32; ++c)
          if (c < dpl) acc[qi][c] = fmaf(pj, Vs[j][lane + 32 * c], acc[qi][c]);
      }
    }
  }

  T* O = static_cast<T*>(a.o) + layer * a.o_sl + head * a.o_sh;
#pragma unroll
  for (int qi = 0; qi < 4; ++qi) {
    const int p = q0 + warp * 4 + qi;
    if (p >= a.Nq) continue;
    const float inv = (l[qi] > 0.f) ? 1.f / l[qi] : 0.f;
#pragma unroll
    for (int c = 0; c < kMaxD / 32; ++c)
      if (c < dpl) O[(int64_t)p * a.o_st + lane + 32 * c] = from_f<T>(acc[qi][c] * inv);
    if (a.lse && lane == 0)
      a.lse[((int64_t)layer * a.H + head) * a.Nq + p] = (l[qi] > 0.f) ? m[qi] + logf(l[qi]) : -INFINITY;
  }
}

bool attn_simt_supported(const AttnArgs& a) { return a.d <= kMaxD && (a.d % 32) == 0; }

cudaError_t launch_attn_simt(const AttnArgs& a, cudaStream_t s) {
  if (!attn_simt_supported(a)) return cudaErrorNotSupported;
  dim3 grid((a.Nq + kQB - 1) / kQB, a.H, a.L);
  if (a.dtype == CRC_F32)
    attn_simt_kernel<float><<<grid, 128, 0, s>>>(a);
  else
    attn_simt_kernel<__nv_bfloat16><<<grid, 128, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace crc
