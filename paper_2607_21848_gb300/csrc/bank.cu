// Memory bank maintenance and the cache update (Sec. 4.2, "Cache layout").
//
// The bank keeps every generated chunk's frames' camera records, its (c_j, v_j)
// pose summary for Eq. 1 and its depth maps for Eq. 4, and its K/V in slab
// j % num_slabs (with the slab's owner recorded when the bank tracks its slabs).  The cache update also writes the new chunk's K/V into the
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
  // chunk index, destinations and frame records: the arguments', or those a step descriptor selects
  int chunk = a.chunk;
  const double* rec = &a.frames.rec[0][0];
  float* depth_dst = a.depth_dst;
  char* slab = a.slab;
  int32_t* owner = a.slab_owner;
  char* win_k = a.win_k;
  char* win_v = a.win_v;
  if (a.step) {
    const int n = a.step->n, woff = a.step->window_offset;
    if (n < 0 || n >= a.capacity || woff < -1 || (woff >= 0 && (int64_t)woff + a.Nc > a.n_keys)) {
      if (blockIdx.x == 0 && tid == 0) atomicExch(a.status, CRC_STEP_BAD_DESCRIPTOR);
      return;
    }
    chunk = n;
    rec = reinterpret_cast<const double*>(a.step->frames);
    depth_dst = a.depth_base + (int64_t)n * a.depth_count;
    if (a.k_src) {
      slab = a.kv_base + (int64_t)(n % a.num_slabs) * a.slab_bytes;
      owner = a.slab_chunk ? a.slab_chunk + n % a.num_slabs : nullptr;
      win_k = woff >= 0 ? a.cache_k + (int64_t)woff * a.win_token_stride : nullptr;
      win_v = woff >= 0 ? a.cache_v + (int64_t)woff * a.win_token_stride : nullptr;
    }
  }
  if (blockIdx.x == 0) {
    const int F = a.frames.F;
    double* dst = a.bank_frames + (size_t)chunk * F * kFrameDoubles;
    for (int i = tid; i < F * kFrameDoubles; i += blockDim.x) dst[i] = rec[i];
    if (tid == 0) {
      if (owner) *owner = chunk;  // the slab now holds this chunk's K/V
      double c[3], v[3];
      chunk_summary(rec, F, c, v);
      for (int e = 0; e < 3; ++e) {
        a.bank_centre[(size_t)chunk * 3 + e] = c[e];
        a.bank_view[(size_t)chunk * 3 + e] = v[e];
      }
    }
  }
  const int gtid = blockIdx.x * blockDim.x + tid;
  const int gthreads = gridDim.x * blockDim.x;
  for (int i = gtid; i < a.depth_count; i += gthreads) depth_dst[i] = a.depth_src[i];
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
    char* dst = slab + kv * half + rem * a.row_bytes;
    if (win_k)
      warp_copy_row<2>(src, dst, (kv ? win_v : win_k) + l * a.win_layer_stride + t * a.win_token_stride, a.row_bytes,
                       lane);
    else
      warp_copy_row<1>(src, dst, nullptr, a.row_bytes, lane);
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
