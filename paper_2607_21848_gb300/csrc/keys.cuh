// Key-column metadata of the segmented cache (Sec. 4.2 cache layout, Sec. 4.3
// design choice ii): whether a key is active, and for keys of a retrieved slot
// the source frame s = slot * F + (position in slot) / (h w) and the key's grid
// position u_k = (x, y) inside that frame.
#pragma once

#include "internal.cuh"

namespace crc {

struct KeyInfo {
  int active;
  int src;    // -1: no bias on this column
  int frame;  // keys of the current chunk (CRC_SEG_CURRENT): their latent frame, else -1
  float x, y;
};

__device__ __forceinline__ KeyInfo key_info_of(const AttnArgs& a, int key) {
  KeyInfo ki{0, -1, -1, 0.f, 0.f};
  if (key >= a.Nk) return ki;
  for (int g = 0; g < a.nseg; ++g) {
    const crc_segment sg = a.seg[g];
    if (key < sg.offset || key >= sg.offset + seg_length(a, g)) continue;
    if (sg.kind == CRC_SEG_RETRIEVED) {
      if (a.slot_chunk && a.slot_chunk[sg.slot] < 0) return ki;  // empty slot: masked
      const int hw = a.h * a.w;
      const int loc = key - sg.offset;
      const int fr = loc / hw;
      const int rem = loc - fr * hw;
      const int row = rem / a.w;
      ki.src = sg.slot * a.F + fr;
      ki.y = (float)row;
      ki.x = (float)(rem - row * a.w);
    } else if (sg.kind == CRC_SEG_CURRENT) {
      ki.frame = (key - sg.offset) / (a.h * a.w);
    }
    ki.active = 1;
    return ki;
  }
  return ki;
}

}  // namespace crc
