// Internal declarations shared by the CUDA translation units of libcrc.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "crc.h"

namespace crc {

// Records e as the calling thread's last CUDA error (crc_last_cuda_error) and
// returns CRC_ERR_CUDA: for entry points defined outside api.cu.
crc_status record_cuda_error(cudaError_t e);

// One crc_frame record is 21 doubles: K[9], R[9], c[3].
constexpr int kFrameDoubles = 21;

struct FrameSet {
  double rec[CRC_MAX_FRAMES][kFrameDoubles];
  int32_t F;
};

// Chunk centre (mean of frame centres) and unit view direction (normalised sum of
// optical axes, R[:, 2]) in fp64 with explicit round-to-nearest operations, so that
// no multiply-add is ever contracted; summation runs in frame order.
__device__ inline void chunk_summary(const double* rec, int F, double c[3], double v[3]) {
  double c0 = rec[18], c1 = rec[19], c2 = rec[20];
  double v0 = rec[9 + 2], v1 = rec[9 + 5], v2 = rec[9 + 8];
  for (int f = 1; f < F; ++f) {
    const double* r = rec + f * kFrameDoubles;
    c0 = __dadd_rn(c0, r[18]);
    c1 = __dadd_rn(c1, r[19]);
    c2 = __dadd_rn(c2, r[20]);
    v0 = __dadd_rn(v0, r[9 + 2]);
    v1 = __dadd_rn(v1, r[9 + 5]);
    v2 = __dadd_rn(v2, r[9 + 8]);
  }
  const double fF = (double)F;
  c[0] = __ddiv_rn(c0, fF);
  c[1] = __ddiv_rn(c1, fF);
  c[2] = __ddiv_rn(c2, fF);
  const double nrm = __dsqrt_rn(__dadd_rn(__dadd_rn(__dmul_rn(v0, v0), __dmul_rn(v1, v1)), __dmul_rn(v2, v2)));
  v[0] = __ddiv_rn(v0, nrm);
  v[1] = __ddiv_rn(v1, nrm);
  v[2] = __ddiv_rn(v2, nrm);
}

// ---- launchers (defined in the kernel translation units) --------------------

struct PoseInsertArgs {
  double* frames;   // bank [capacity][F][21]
  double* centre;   // bank [capacity][3]
  double* view;     // bank [capacity][3]
  int32_t F;
  int32_t first;
  int32_t count;
};
cudaError_t launch_pose_summary(const PoseInsertArgs& a, cudaStream_t s);

// Per-step values of crc_chunk_step, read on the device.  A launcher given a step
// takes the chunk index, window offset, fallback chunk, re-positioning target,
// segment lengths and frames from it instead of its own arguments.
using StepDesc = crc_step;
static_assert(sizeof(crc_frame) == 21 * sizeof(double), "crc_frame is 21 packed doubles");

struct CacheUpdateArgs {
  const StepDesc* step;    // crc_chunk_step: chunk, window offset, frames and the pointers below
  int32_t* status;         // set to CRC_STEP_BAD_DESCRIPTOR for a descriptor out of range
  int32_t capacity;        // bank chunks (descriptor check)
  int32_t num_slabs;
  int64_t slab_bytes;
  char* kv_base;           // bank->kv
  int32_t* slab_chunk;     // bank->slab_chunk or null
  float* depth_base;       // bank->depth
  char* cache_k;           // cache bases (window slot derived from the descriptor)
  char* cache_v;
  int32_t n_keys;
  FrameSet frames;
  double* bank_frames;
  double* bank_centre;
  double* bank_view;
  int32_t* slab_owner;     // bank->slab_chunk + chunk % num_slabs, or null
  int32_t chunk;
  const float* depth_src;  // [F][h][w]
  float* depth_dst;        // bank depth + chunk * F*h*w
  int32_t depth_count;
  const char* k_src;       // [L][Nc][H][d] dense, or null
  const char* v_src;
  char* slab;              // bank kv slab of this chunk: [2][L][Nc][H][d]
  char* win_k;             // cache k + window offset rows (layer 0), or null
  char* win_v;
  int64_t win_layer_stride;  // bytes
  int64_t win_token_stride;  // bytes
  int32_t L;
  int32_t Nc;
  int32_t row_bytes;       // H*d*elem
};
cudaError_t launch_cache_update(const CacheUpdateArgs& a, cudaStream_t s);

// Slab-to-cache gather of the retrieved slots, with the optional temporal RoPE
// re-positioning of the keys (crc_rope).
struct GatherArgs {
  const char* pool;     // [num_slabs][2][L][Nc][H][d]; null disables the gather
  int32_t num_slabs;
  int64_t slab_bytes;
  int64_t kv_bytes;     // bytes of the K half of a slab
  char* cache_k;
  char* cache_v;
  int64_t cache_layer_stride;  // bytes
  int64_t cache_token_stride;  // bytes
  int32_t slot_offset[CRC_MAX_K];  // token offset of slot r's segment, -1 if none
  int32_t L;
  int32_t Nc;
  int32_t row_bytes;    // H*d*elem
  int32_t d;            // head dim
  int32_t elem_bytes;   // 2 (bf16) or 4 (fp32)
  int32_t F;
  const StepDesc* step;  // crc_chunk_step: rope_pos_slot0 from the descriptor
  // rope (rope_pairs = 0: plain copy)
  int32_t rope_pairs, rope_c0, rope_interleaved;
  int32_t rope_pos_slot0, rope_pos_stride, rope_frame_pos0;
  double rope_omega[CRC_MAX_ROPE_PAIRS];  // theta^(-i/pairs)
};

// One candidate of the top-k: the score as an order-preserving 64-bit key, and j.
struct TopkCand {
  unsigned long long key;
  int32_t j;
  int32_t pad;
};

struct RetrieveArgs {
  const StepDesc* step;  // crc_chunk_step: n, count = n + 1, ext_first and frames from the descriptor
  int32_t* status;       // descriptor check (with a step)
  int32_t capacity;
  FrameSet cur;
  const double* centre;
  const double* view;
  const int32_t* slab_chunk;  // [num_slabs] chunk held by each K/V slab, or null (no residency test)
  int32_t num_slabs;
  int32_t count;
  int32_t n;
  double E, w_v, tau_c, cos_tau_v;
  int32_t delta, k, ext_first, ext_min, exclude_sink;
  int32_t* d_idx;
  double* d_score;
  int32_t* d_count;
  TopkCand* partial;     // [grid][k] per-block candidates (workspace; null with one block)
  unsigned int* ticket;  // blocks done (workspace; zeroed before the launch)
};

// Blocks and workspace bytes of the top-k launch over `count` bank entries.
int retrieve_blocks(int32_t count);
size_t retrieve_workspace_bytes(int32_t count, int32_t k);

struct GatherOnlyArgs {
  const int32_t* d_idx;  // [k] chunk per slot (negative = empty)
  int32_t k;
  GatherArgs g;
};
// The top-k launch, then (g.pool non-null) the gather launch that reads its d_idx.
cudaError_t launch_retrieve(const RetrieveArgs& a, const GatherArgs& g, cudaStream_t s);
cudaError_t launch_gather(const GatherOnlyArgs& a, cudaStream_t s, bool after_topk = false);

struct CorrespondArgs {
  const StepDesc* step;      // crc_chunk_step: the current frames from the descriptor
  FrameSet cur;
  const float* depth;        // [F][h][w]
  const double* bank_frames; // [capacity][F][21]
  const float* bank_depth;   // [capacity][F][h][w]
  int32_t capacity;
  const int32_t* d_idx;
  const int32_t* d_count;    // may be null
  int32_t k, F, h, w;
  float eps;                 // +inf disables Eq. 4
  float* uv;
  int32_t* cell;             // may be null
  uint8_t* valid;
};
cudaError_t launch_correspond(const CorrespondArgs& a, cudaStream_t s);

struct AttnArgs {
  const StepDesc* step;  // crc_chunk_step: segment lengths from the descriptor (at most seg[].length)
  const void* q;
  const void* k;
  const void* v;
  void* o;
  float* lse;
  int64_t q_sl, q_st, q_sh;   // element strides
  int64_t k_sl, k_st, k_sh;
  int64_t o_sl, o_st, o_sh;
  int32_t L, H, d, Nq, Nk;
  int32_t F, h, w, S;
  int32_t nseg;
  crc_segment seg[CRC_MAX_SEGMENTS];
  const float* uv;
  const uint8_t* valid;
  const int32_t* slot_chunk;
  float lambda;
  float sigma;
  int32_t dtype;
  int32_t* status;
  int32_t bias_form;  // 0: Eq. 2 quadratic; 1: additive Gaussian (CRC_ATTN_GAUSSIAN)
  int32_t bias_direct;  // Eq. 2 evaluated per score even where the tensor-core expansion is accurate
  int32_t frame_causal; // CRC_ATTN_FRAME_CAUSAL: later frames of the CURRENT segment are masked per query
  int32_t skip_far;   // CRC_ATTN_SKIP_FAR in force (tensor-core kernel)
  float skip_d2;      // squared grid distance beyond which a retrieved tile is skipped
};
// Length of cache segment g in this call: the descriptor's, clamped to the plan's.
// A retrieved or current-chunk segment is all or nothing (N_c keys or none).
__device__ __forceinline__ int32_t seg_length(const AttnArgs& a, int g) {
  const int32_t len = a.seg[g].length;
  if (a.step == nullptr) return len;
  const int32_t sl = a.step->seg_length[g];
  if (a.seg[g].kind == CRC_SEG_RETRIEVED || a.seg[g].kind == CRC_SEG_CURRENT) return sl > 0 ? len : 0;
  return sl < 0 ? 0 : (sl < len ? sl : len);
}

cudaError_t launch_attn_simt(const AttnArgs& a, cudaStream_t s);
cudaError_t launch_attn_tc(const AttnArgs& a, cudaStream_t s);
// Whether a kernel can take these arguments (checked on the host before any launch).
bool attn_simt_supported(const AttnArgs& a);
bool attn_tc_supported(const AttnArgs& a);
// Error bound of the tensor-core expansion of Eq. 2, in base-2 logit units, and the
// bound above which the tensor-core kernel evaluates Eq. 2 per score instead.
double bias_expansion_bound(float lambda, float sigma, int h, int w);
constexpr double kExpansionLimit = 0x1p-9;

}  // namespace crc
