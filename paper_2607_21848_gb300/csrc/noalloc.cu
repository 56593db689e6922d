// crc_retrieve_noalloc: the retrieval for callers that cannot allocate device memory.
//
// crc_retrieve needs a workspace for banks of more than 512 entries, where several
// blocks score the bank and meet to merge their candidates.  Some callers cannot
// allocate one: an engine's render thread with a fixed per-frame budget (cudaMalloc
// and cudaFree can synchronise the device and take milliseconds), a plugin whose host
// application owns every byte of GPU memory, or a stream that must not fail with an
// out-of-memory error half-way through.  This entry point uses a fixed scratch array
// that lives in the library's own device memory instead, loaded with the library and
// held by every GPU that loads it until the process exits.
#include <mutex>

#include "internal.cuh"

namespace {

// The fixed scratch: per-block top-k candidates and the blocks' completion ticket.
static __device__ __align__(256) unsigned char g_retrieve_scratch[CRC_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device, looked up once per device.
// (In host code the array's name stands for a host-side shadow, not a device address.)
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (g_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_retrieve_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return cudaSuccess;
}

}  // namespace

extern "C" crc_status crc_retrieve_noalloc(const crc_bank* bank, int32_t bank_count, const crc_shape* shape,
                                           const crc_frame* cur, int32_t n, const crc_retrieval* p,
                                           const crc_cache* cache, const crc_rope* rope, int32_t* d_idx,
                                           double* d_score, int32_t* d_count, cudaStream_t s) {
  if (!p) return CRC_ERR_INVALID_ARG;
  // crc_retrieve checks everything else; a size of 0 means no scratch is needed
  const size_t need = crc_retrieve_workspace_size(bank_count, p->k);
  if (need > CRC_NOALLOC_SCRATCH_BYTES) return CRC_ERR_TOO_LARGE;
  void* scratch = nullptr;
  if (need > 0) {
    const cudaError_t e = scratch_address(&scratch);
    if (e != cudaSuccess) return crc::record_cuda_error(e);
  }
  return crc_retrieve(bank, bank_count, shape, cur, n, p, cache, rope, d_idx, d_score, d_count, scratch,
                      need > 0 ? (size_t)CRC_NOALLOC_SCRATCH_BYTES : 0, s);
}
