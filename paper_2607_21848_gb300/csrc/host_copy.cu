// crc_host_copy: copies between page-locked host memory and device memory issued by
// the SMs over the coherent CPU-GPU link, instead of by the copy engines.
//
// On Grace-Blackwell the GPU reaches page-locked host memory directly: a kernel's
// 16-byte loads and stores move host data at the link's own rate (about 210 GB/s
// host-to-device and 190 GB/s device-to-host measured on GB300), and a handful of
// SMs suffice for that rate.  The copy engines reach the same rate, but on some
// machines they stall for tens of milliseconds at a time, with or without other
// work on the GPU; copies issued by the SMs were not seen to stall.
#include "internal.cuh"

namespace {

constexpr int kCopyThreads = 1024;
constexpr int kCopyInFlight = 4;  // independent 16-byte loads per thread before its stores
constexpr int kCopyDefaultBlocks = 8;

// Every thread moves kCopyInFlight vectors per round, strided by the grid, so each
// warp's accesses are contiguous 512-byte runs.  Loads are cached in L2 only and
// stores are streaming: the data passes through once.  (Beside the attention kernel
// this form moved 1.72 GB of step inputs and output in 10.2 ms; the same loop with
// plain loads and stores, compiled with fewer loads in flight, took 14.5 ms.)
// Block 0 copies the byte tail first.
__global__ void __launch_bounds__(kCopyThreads, 1)
    host_copy_kernel(const uint4* __restrict__ src, uint4* __restrict__ dst, size_t n,
                     const unsigned char* __restrict__ src_tail, unsigned char* __restrict__ dst_tail, int tail) {
  if (blockIdx.x == 0 && (int)threadIdx.x < tail) dst_tail[threadIdx.x] = src_tail[threadIdx.x];
  const size_t stride = (size_t)gridDim.x * blockDim.x;
  size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
  for (; i + (kCopyInFlight - 1) * stride < n; i += kCopyInFlight * stride) {
    uint4 r[kCopyInFlight];
#pragma unroll
    for (int u = 0; u < kCopyInFlight; ++u) r[u] = __ldcg(src + i + u * stride);
#pragma unroll
    for (int u = 0; u < kCopyInFlight; ++u) __stcs(dst + i + u * stride, r[u]);
  }
  for (; i < n; i += stride) __stcs(dst + i, __ldcg(src + i));
}

// The device address of [p, p + bytes) if the current device can reach all of it:
// device memory of this device, page-locked host memory or managed memory, with its
// first and last byte in one contiguous mapping.
crc_status reachable(const void* p, size_t bytes, uintptr_t* dev) {
  int cur = 0;
  cudaError_t e = cudaGetDevice(&cur);
  if (e != cudaSuccess) return crc::record_cuda_error(e);
  cudaPointerAttributes a[2];
  const void* ends[2] = {p, (const unsigned char*)p + (bytes - 1)};
  for (int j = 0; j < 2; ++j) {
    e = cudaPointerGetAttributes(&a[j], ends[j]);
    if (e != cudaSuccess) {
      (void)cudaGetLastError();  // an unknown pointer is an argument error, not a sticky CUDA one
      return CRC_ERR_INVALID_ARG;
    }
    const bool ok = (a[j].type == cudaMemoryTypeDevice && a[j].device == cur) || a[j].type == cudaMemoryTypeHost ||
                    a[j].type == cudaMemoryTypeManaged;
    if (!ok || a[j].devicePointer == nullptr) return CRC_ERR_INVALID_ARG;
  }
  if (a[0].type != a[1].type) return CRC_ERR_INVALID_ARG;
  const uintptr_t d0 = (uintptr_t)a[0].devicePointer, d1 = (uintptr_t)a[1].devicePointer;
  if (d1 < d0 || d1 - d0 != bytes - 1) return CRC_ERR_INVALID_ARG;
  *dev = d0;
  return CRC_OK;
}

}  // namespace

extern "C" crc_status crc_host_copy(void* dst, const void* src, size_t bytes, int32_t blocks, cudaStream_t s) {
  if (bytes == 0) return CRC_OK;
  if (!dst || !src || blocks < 0 || blocks > 4096) return CRC_ERR_INVALID_ARG;
  if (((uintptr_t)dst & 15u) || ((uintptr_t)src & 15u)) return CRC_ERR_UNSUPPORTED;
  uintptr_t d_src = 0, d_dst = 0;
  crc_status st = reachable(src, bytes, &d_src);
  if (st) return st;
  if ((st = reachable(dst, bytes, &d_dst))) return st;
  if (d_src < d_dst + bytes && d_dst < d_src + bytes) return CRC_ERR_INVALID_ARG;  // overlapping ranges
  const size_t n = bytes / 16;
  const int tail = (int)(bytes % 16);
  int grid = blocks > 0 ? blocks : kCopyDefaultBlocks;
  // no more blocks than there are vectors to move (at least one, for the tail)
  const size_t per_block = (size_t)kCopyThreads;
  if ((size_t)grid * per_block > n) grid = (int)((n + per_block - 1) / per_block);
  if (grid < 1) grid = 1;
  host_copy_kernel<<<grid, kCopyThreads, 0, s>>>((const uint4*)d_src, (uint4*)d_dst, n,
                                                 (const unsigned char*)(d_src + n * 16),
                                                 (unsigned char*)(d_dst + n * 16), tail);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? CRC_OK : crc::record_cuda_error(e);
}
