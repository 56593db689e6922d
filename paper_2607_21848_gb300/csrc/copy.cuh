// Warp-cooperative row copies used by the cache update and the retrieval gather.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace crc {

// Copy `bytes` (a multiple of 16) from src to up to two destinations with 16-byte
// vector accesses; each lane keeps four loads in flight before storing.
__device__ __forceinline__ void warp_copy_row(const char* __restrict__ src, char* __restrict__ dst0,
                                              char* __restrict__ dst1, int bytes, int lane) {
  const uint4* s = reinterpret_cast<const uint4*>(src);
  uint4* d0 = reinterpret_cast<uint4*>(dst0);
  uint4* d1 = reinterpret_cast<uint4*>(dst1);
  const int n = bytes >> 4;
  int c = lane;
  for (; c + 96 < n; c += 128) {
    uint4 a0 = __ldg(s + c), a1 = __ldg(s + c + 32), a2 = __ldg(s + c + 64), a3 = __ldg(s + c + 96);
    d0[c] = a0; d0[c + 32] = a1; d0[c + 64] = a2; d0[c + 96] = a3;
    if (d1) { d1[c] = a0; d1[c + 32] = a1; d1[c + 64] = a2; d1[c + 96] = a3; }
  }
  for (; c < n; c += 32) {
    uint4 a0 = __ldg(s + c);
    d0[c] = a0;
    if (d1) d1[c] = a0;
  }
}

}  // namespace crc
