// Depth-reprojection correspondence (Sec. 4.3, Eq. 3) with the occlusion-aware
// visibility test (Eq. 4) and the exact-fallback rules of the design choices.
//
// One thread per (query token p, source frame s) pair, pairs laid out [N_q][S] so
// that every output array is written fully coalesced.  At block start the
// per-(target frame t, source frame s) transform
//     A_ts = R_s^T R_t K_t^-1,   b_ts = R_s^T (c_t - c_s),   K_s
// is composed from the current frames (kernel argument) and the bank records of
// the retrieved chunk d_idx[r] (device memory, so no host round trip) and kept in
// shared memory.  The composition runs in fp32 -- the per-pair arithmetic that
// consumes it is fp32 anyway -- except for the camera-centre difference, which is
// formed in fp64 so that nearby centres do not cancel; fp64 throughput on this GPU
// is a small fraction of fp32's and every block repeats the composition.  Per pair:
//     X_s = z_p A_ts (j, i, 1)^T + b_ts  (= Eq. 3's X_s),   u^ = pi(K_s X_s).
#include <math.h>

#include "internal.cuh"

namespace crc {

namespace {

constexpr int kMaxS = CRC_MAX_K * CRC_MAX_FRAMES;
constexpr int kMaxPairs = CRC_MAX_FRAMES * kMaxS;

// 24 words, 16-byte aligned, so that a pair's transform is six vector loads
struct __align__(16) PairXf {
  float A[9];
  float b[3];
  float Ks[9];
  int depth_off;  // offset of D_s in the bank depth array, -1 if the pair is not a retrieval
  int pad[2];
};

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

__global__ void __launch_bounds__(256) correspond_kernel(const __grid_constant__ CorrespondArgs a) {
  __shared__ PairXf px[kMaxPairs];
  const int S = a.k * a.F;
  const int npairs = a.F * S;
  const int hw = a.h * a.w;
  for (int q = threadIdx.x; q < npairs; q += blockDim.x) {
    const int t = q / S, s = q - (q / S) * S;
    const int r = s / a.F, f = s - (s / a.F) * a.F;
    const int j = a.d_idx[r];
    bool ok = (j >= 0) && (j < a.capacity);
    if (a.d_count) ok = ok && (r < *a.d_count);
    PairXf x;
    x.pad[0] = x.pad[1] = 0;
    if (ok) {
      const double* ft = &a.cur.rec[t][0];
      const double* fs = a.bank_frames + ((size_t)j * a.F + f) * kFrameDoubles;
      float Kt[9], Rt[9], Rs[9], Ki[9], RK[9];
      for (int e = 0; e < 9; ++e) {
        Kt[e] = (float)ft[e];
        Rt[e] = (float)ft[9 + e];
        Rs[e] = (float)fs[9 + e];
      }
      mat3_inverse(Kt, Ki);
      for (int m = 0; m < 3; ++m)
        for (int n = 0; n < 3; ++n) RK[3 * m + n] = Rt[3 * m + 0] * Ki[n] + Rt[3 * m + 1] * Ki[3 + n] + Rt[3 * m + 2] * Ki[6 + n];
      // A = R_s^T (R_t K_t^-1)
      for (int m = 0; m < 3; ++m)
        for (int n = 0; n < 3; ++n) x.A[3 * m + n] = Rs[m] * RK[n] + Rs[3 + m] * RK[3 + n] + Rs[6 + m] * RK[6 + n];
      const float dc[3] = {(float)(ft[18] - fs[18]), (float)(ft[19] - fs[19]), (float)(ft[20] - fs[20])};
      for (int m = 0; m < 3; ++m) x.b[m] = Rs[m] * dc[0] + Rs[3 + m] * dc[1] + Rs[6 + m] * dc[2];
      for (int e = 0; e < 9; ++e) x.Ks[e] = (float)fs[e];
      x.depth_off = (int)(((size_t)j * a.F + f) * hw);
    } else {
      for (int e = 0; e < 9; ++e) x.A[e] = x.Ks[e] = 0.f;
      x.b[0] = x.b[1] = x.b[2] = 0.f;
      x.depth_off = -1;
    }
    px[q] = x;
  }
  __syncthreads();

  const int total = a.F * hw * S;
  const bool vis_test = !isinf(a.eps);
  const float one_eps = 1.0f + a.eps;
  // The block size is a multiple of S, so the grid stride is too and each thread
  // keeps one source frame s for all its pairs.  Its transform for target frame t
  // stays in registers and is reloaded only when t changes (at most F times).
  // Each thread carries kILP pairs at once, so that their query-depth loads and
  // then their source-depth gathers overlap in flight.
  constexpr int kILP = 4;
  const int stride = gridDim.x * blockDim.x;
  const int first = blockIdx.x * blockDim.x + threadIdx.x;
  const int s_own = first - (int)fastdiv((uint32_t)first, a.div_S) * S;
  int t_cached = -1;
  PairXf x;
  for (int base = first; base < total; base += kILP * stride) {
    int pr[kILP], tr[kILP], jx[kILP], iy[kILP];
    float z[kILP];
#pragma unroll
    for (int u = 0; u < kILP; ++u) {
      const int idx = base + u * stride;
      pr[u] = idx < total ? (int)fastdiv((uint32_t)idx, a.div_S) : -1;
      tr[u] = -1;
      z[u] = 0.f;
      if (pr[u] >= 0) {
        tr[u] = (int)fastdiv((uint32_t)pr[u], a.div_hw);
        const int rem = pr[u] - tr[u] * hw;
        iy[u] = (int)fastdiv((uint32_t)rem, a.div_w);
        jx[u] = rem - iy[u] * a.w;
        z[u] = a.depth[pr[u]];
      }
    }
    float ux[kILP], uy[kILP], X2[kILP];
    int cell[kILP], doff[kILP];
    bool valid[kILP];
#pragma unroll
    for (int u = 0; u < kILP; ++u) {
      ux[u] = uy[u] = __int_as_float(0x7fc00000);  // NaN when the pair is not a retrieval
      valid[u] = false;
      cell[u] = -1;
      X2[u] = 0.f;
      doff[u] = -1;
      if (pr[u] < 0) continue;
      if (tr[u] != t_cached) {
#pragma unroll
        for (int v = 0; v < 6; ++v)
          reinterpret_cast<float4*>(&x)[v] = reinterpret_cast<const float4*>(&px[tr[u] * S + s_own])[v];
        t_cached = tr[u];
      }
      doff[u] = x.depth_off;
      if (x.depth_off < 0) continue;
      const float u0 = (float)jx[u], u1 = (float)iy[u];
      const float a0 = x.A[0] * u0 + x.A[1] * u1 + x.A[2];
      const float a1 = x.A[3] * u0 + x.A[4] * u1 + x.A[5];
      const float a2 = x.A[6] * u0 + x.A[7] * u1 + x.A[8];
      const float X0 = z[u] * a0 + x.b[0];
      const float X1 = z[u] * a1 + x.b[1];
      X2[u] = z[u] * a2 + x.b[2];
      const float q0 = x.Ks[0] * X0 + x.Ks[1] * X1 + x.Ks[2] * X2[u];
      const float q1 = x.Ks[3] * X0 + x.Ks[4] * X1 + x.Ks[5] * X2[u];
      const float q2 = x.Ks[6] * X0 + x.Ks[7] * X1 + x.Ks[8] * X2[u];
      const float iq = 1.0f / q2;  // one division: u^ within an ulp of q0 / q2
      ux[u] = q0 * iq;
      uy[u] = q1 * iq;
      const float fx = floorf(ux[u] + 0.5f), fy = floorf(uy[u] + 0.5f);
      valid[u] = isfinite(z[u]) && z[u] > 0.f && isfinite(ux[u]) && isfinite(uy[u]) && X2[u] > 0.f && fx >= 0.f &&
                 fx < (float)a.w && fy >= 0.f && fy < (float)a.h;
      if (valid[u]) cell[u] = (int)fy * a.w + (int)fx;
    }
    float ds[kILP];
#pragma unroll
    for (int u = 0; u < kILP; ++u)
      ds[u] = (vis_test && valid[u]) ? a.bank_depth[doff[u] + cell[u]] : 0.f;
#pragma unroll
    for (int u = 0; u < kILP; ++u) {
      if (pr[u] < 0) continue;
      if (vis_test && valid[u] && !(X2[u] <= one_eps * ds[u])) {
        valid[u] = false;
        cell[u] = -1;
      }
      const int idx = base + u * stride;
      reinterpret_cast<float2*>(a.uv)[idx] = make_float2(ux[u], uy[u]);
      if (a.cell) a.cell[idx] = cell[u];
      a.valid[idx] = valid[u] ? 1 : 0;
    }
  }
}

cudaError_t launch_correspond(const CorrespondArgs& a, cudaStream_t s) {
  const int total = a.F * a.h * a.w * a.k * a.F;
  if (total == 0) return cudaSuccess;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  // grid-stride over the pairs with four pairs in flight per thread: one resident
  // wave, so that each block's composition of the transforms is amortised over
  // many pairs
  const int S = a.k * a.F;
  const int threads = (256 / S) * S;  // a multiple of S (S <= 32)
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, correspond_kernel, threads, 0) != cudaSuccess ||
      per_sm < 1)
    per_sm = 1;
  int blocks = (total + 4 * threads - 1) / (4 * threads);
  if (blocks > per_sm * sms) blocks = per_sm * sms;
  correspond_kernel<<<blocks, threads, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace crc
