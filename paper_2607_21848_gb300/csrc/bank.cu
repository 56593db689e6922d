// Memory bank maintenance and the cache update (Sec. 4.2, "Cache layout").
//
// The bank keeps every generated chunk retrievable: its frames' camera records,
// its (c_j, v_j) pose summary for Eq. 1, its depth maps for Eq. 4, and its K/V in
// slab j % num_slabs.  The cache update also writes the new chunk's K/V into the
// recent-window slot chosen by the caller; the anchor (sink) is never touched.
#include "copy.cuh"
#include "internal.cuh"

namespace crc {

__global__ void pose_summary_kernel(PoseInsertArgs a) {
  const int j = blockIdx.x * blockDim.x + threadIdx.x;
  if (j >= a.count) return;
  const int chunk = a.first + j;
  const double* rec = a.frames + (size_t)chunk * a.F * kFrameDoubles;
  double c[3], v[3];
  chunk_summary(rec, a.F, c, v);
  for (int e = 0; e < 3; ++e) {
    a.centre[(size_t)chunk * 3 + e] = c[e];
    a.view[(size_t)chunk * 3 + e] = v[e];
  }
}

cudaError_t launch_pose_summary(const PoseInsertArgs& a, cudaStream_t s) {
  if (a.count == 0) return cudaSuccess;
  const int threads = 128;
  pose_summary_kernel<<<(a.count + threads - 1) / threads, threads, 0, s>>>(a);
  return cudaGetLastError();
}

__global__ void __launch_bounds__(256) cache_update_kernel(const __grid_constant__ CacheUpdateArgs a) {
  const int tid = threadIdx.x;
  if (blockIdx.x == 0) {
    const int F = a.frames.F;
    double* dst = a.bank_frames + (size_t)a.chunk * F * kFrameDoubles;
    for (int i = tid; i < F * kFrameDoubles; i += blockDim.x) dst[i] = a.frames.rec[i / kFrameDoubles][i % kFrameDoubles];
    if (tid == 0) {
      double c[3], v[3];
      chunk_summary(&a.frames.rec[0][0], F, c, v);
      for (int e = 0; e < 3; ++e) {
        a.bank_centre[(size_t)a.chunk * 3 + e] = c[e];
        a.bank_view[(size_t)a.chunk * 3 + e] = v[e];
      }
    }
  }
  const int gtid = blockIdx.x * blockDim.x + tid;
  const int gthreads = gridDim.x * blockDim.x;
  for (int i = gtid; i < a.depth_count; i += gthreads) a.depth_dst[i] = a.depth_src[i];
  if (a.k_src == nullptr) return;

  // one warp per token row of H*d elements; rows ordered (kv, layer, token)
  const int lane = tid & 31;
  const int gwarp = gtid >> 5;
  const int nwarps = gthreads >> 5;
  const int64_t rows_per_kv = (int64_t)a.L * a.Nc;
  const int64_t half = rows_per_kv * a.row_bytes;
  for (int64_t row = gwarp; row < 2 * rows_per_kv; row += nwarps) {
    const int kv = (int)(row / rows_per_kv);
    const int64_t rem = row - kv * rows_per_kv;
    const int l = (int)(rem / a.Nc);
    const int t = (int)(rem - (int64_t)l * a.Nc);
    const char* src = (kv ? a.v_src : a.k_src) + rem * a.row_bytes;
    char* slab = a.slab + kv * half + rem * a.row_bytes;
    char* win = nullptr;
    if (a.win_k) win = (kv ? a.win_v : a.win_k) + l * a.win_layer_stride + t * a.win_token_stride;
    warp_copy_row(src, slab, win, a.row_bytes, lane);
  }
}

cudaError_t launch_cache_update(const CacheUpdateArgs& a, cudaStream_t s) {
  int blocks = 1;
  if (a.k_src) {
    const int64_t rows = 2LL * a.L * a.Nc;
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t want = (rows + 7) / 8;  // 8 warps per block
    blocks = (int)(want < (int64_t)sms * 4 ? want : (int64_t)sms * 4);
    if (blocks < 1) blocks = 1;
  } else {
    blocks = (a.depth_count + 255) / 256;
    if (blocks < 1) blocks = 1;
  }
  cache_update_kernel<<<blocks, 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace crc
