// Depth-reprojection correspondence (Sec. 4.3, Eq. 3) with the occlusion-aware
// visibility test (Eq. 4) and the exact-fallback rules of the design choices.
//
// One thread per (query token p, source frame s) pair, pairs laid out [N_q][S] so
// that every output array is written fully coalesced.  At block start the
// per-(target frame t, source frame s) transform
//     A_ts = R_s^T R_t K_t^-1,   b_ts = R_s^T (c_t - c_s),   K_s
// is composed in fp64 from the current frames (kernel argument) and the bank
// records of the retrieved chunk d_idx[r] (device memory, so no host round trip)
// and kept in shared memory as fp32.  Per pair:
//     X_s = z_p A_ts (j, i, 1)^T + b_ts  (= Eq. 3's X_s),   u^ = pi(K_s X_s).
#include <math.h>

#include "internal.cuh"

namespace crc {

namespace {

constexpr int kMaxS = CRC_MAX_K * CRC_MAX_FRAMES;
constexpr int kMaxPairs = CRC_MAX_FRAMES * kMaxS;

struct PairXf {
  float A[9];
  float b[3];
  float Ks[9];
  int depth_off;  // offset of D_s in the bank depth array, -1 if the pair is not a retrieval
};

__device__ void mat3_inverse(const double* m, double* inv) {
  const double c00 = m[4] * m[8] - m[5] * m[7];
  const double c01 = m[5] * m[6] - m[3] * m[8];
  const double c02 = m[3] * m[7] - m[4] * m[6];
  const double det = m[0] * c00 + m[1] * c01 + m[2] * c02;
  const double id = 1.0 / det;
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
    if (ok) {
      const double* ft = &a.cur.rec[t][0];
      const double* fs = a.bank_frames + ((size_t)j * a.F + f) * kFrameDoubles;
      double Ki[9], RK[9], A[9];
      mat3_inverse(ft, Ki);
      const double* Rt = ft + 9;
      const double* Rs = fs + 9;
      for (int m = 0; m < 3; ++m)
        for (int n = 0; n < 3; ++n) RK[3 * m + n] = Rt[3 * m + 0] * Ki[n] + Rt[3 * m + 1] * Ki[3 + n] + Rt[3 * m + 2] * Ki[6 + n];
      // A = R_s^T (R_t K_t^-1)
      for (int m = 0; m < 3; ++m)
        for (int n = 0; n < 3; ++n) A[3 * m + n] = Rs[m] * RK[n] + Rs[3 + m] * RK[3 + n] + Rs[6 + m] * RK[6 + n];
      const double dc[3] = {ft[18] - fs[18], ft[19] - fs[19], ft[20] - fs[20]};
      for (int m = 0; m < 3; ++m) x.b[m] = (float)(Rs[m] * dc[0] + Rs[3 + m] * dc[1] + Rs[6 + m] * dc[2]);
      for (int e = 0; e < 9; ++e) {
        x.A[e] = (float)A[e];
        x.Ks[e] = (float)fs[e];
      }
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
  for (int idx = blockIdx.x * blockDim.x + threadIdx.x; idx < total; idx += gridDim.x * blockDim.x) {
    const int p = idx / S;
    const int s = idx - p * S;
    const int t = p / hw;
    const int rem = p - t * hw;
    const int i = rem / a.w;
    const int jx = rem - i * a.w;
    const PairXf& x = px[t * S + s];
    float ux = __int_as_float(0x7fc00000), uy = ux;  // NaN when the pair is not a retrieval
    bool valid = false;
    int cell = -1;
    if (x.depth_off >= 0) {
      const float z = a.depth[p];
      const float u0 = (float)jx, u1 = (float)i;
      const float a0 = x.A[0] * u0 + x.A[1] * u1 + x.A[2];
      const float a1 = x.A[3] * u0 + x.A[4] * u1 + x.A[5];
      const float a2 = x.A[6] * u0 + x.A[7] * u1 + x.A[8];
      const float X0 = z * a0 + x.b[0];
      const float X1 = z * a1 + x.b[1];
      const float X2 = z * a2 + x.b[2];
      const float q0 = x.Ks[0] * X0 + x.Ks[1] * X1 + x.Ks[2] * X2;
      const float q1 = x.Ks[3] * X0 + x.Ks[4] * X1 + x.Ks[5] * X2;
      const float q2 = x.Ks[6] * X0 + x.Ks[7] * X1 + x.Ks[8] * X2;
      ux = q0 / q2;
      uy = q1 / q2;
      const float fx = floorf(ux + 0.5f), fy = floorf(uy + 0.5f);
      valid = isfinite(z) && z > 0.f && isfinite(ux) && isfinite(uy) && X2 > 0.f && fx >= 0.f &&
              fx < (float)a.w && fy >= 0.f && fy < (float)a.h;
      if (valid) {
        const int cx = (int)fx, cy = (int)fy;
        if (vis_test) valid = X2 <= one_eps * a.bank_depth[x.depth_off + cy * a.w + cx];
        if (valid) cell = cy * a.w + cx;
      }
    }
    reinterpret_cast<float2*>(a.uv)[idx] = make_float2(ux, uy);
    if (a.cell) a.cell[idx] = cell;
    a.valid[idx] = valid ? 1 : 0;
  }
}

cudaError_t launch_correspond(const CorrespondArgs& a, cudaStream_t s) {
  const int total = a.F * a.h * a.w * a.k * a.F;
  if (total == 0) return cudaSuccess;
  int blocks = (total + 255) / 256;
  if (blocks > 4096) blocks = 4096;
  correspond_kernel<<<blocks, 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace crc
