// C ABI entry points: host-side argument validation, then one kernel launch each.
#include <math.h>
#include <string.h>

#include "internal.cuh"

// Build with -DCRC_NVTX (CRC_NVTX=1 in the environment of the build script) to wrap
// every entry point in an NVTX range, for timeline tools.
#ifdef CRC_NVTX
#include <nvtx3/nvToolsExt.h>
namespace {
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
};
}  // namespace
#define CRC_RANGE(name) NvtxRange crc_nvtx_range_(name)
#else
#define CRC_RANGE(name) \
  do {                  \
  } while (0)
#endif

namespace {

thread_local int32_t g_last_cuda_error = 0;

crc_status cuda_fail(cudaError_t e) {
  g_last_cuda_error = (int32_t)e;
  return CRC_ERR_CUDA;
}

int elem_bytes(int32_t dtype) { return dtype == CRC_BF16 ? 2 : 4; }

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

crc_status check_shape(const crc_shape* sh) {
  if (!sh) return CRC_ERR_INVALID_ARG;
  if (sh->L < 1 || sh->H < 1 || sh->F < 1 || sh->F > CRC_MAX_FRAMES || sh->h < 1 || sh->w < 1)
    return CRC_ERR_INVALID_ARG;
  if (sh->dtype != CRC_F32 && sh->dtype != CRC_BF16) return CRC_ERR_UNSUPPORTED;
  if (sh->d < 8 || (sh->d % 8) != 0) return CRC_ERR_UNSUPPORTED;
  const int64_t nc = (int64_t)sh->F * sh->h * sh->w;
  if (nc > (1 << 24)) return CRC_ERR_SHAPE;
  return CRC_OK;
}

bool frames_ok(const crc_frame* fr, int F) {
  for (int f = 0; f < F; ++f) {
    const double* K = fr[f].K;
    if (K[6] != 0.0 || K[7] != 0.0 || K[8] != 1.0) return false;
    for (int e = 0; e < 9; ++e)
      if (!isfinite(fr[f].K[e]) || !isfinite(fr[f].R[e])) return false;
    for (int e = 0; e < 3; ++e)
      if (!isfinite(fr[f].c[e])) return false;
  }
  return true;
}

crc_status check_bank(const crc_bank* b, bool need_kv) {
  if (!b || b->capacity < 1 || !b->frames || !b->centre || !b->view || !b->depth) return CRC_ERR_INVALID_ARG;
  if ((need_kv || b->slab_chunk) && (!b->kv || b->num_slabs < 1)) return CRC_ERR_INVALID_ARG;
  return CRC_OK;
}

// The cache must hold whole token rows of H*d contiguous elements (stride_head = d,
// stride_token >= H*d) with 16-byte aligned rows; k and v share strides.
crc_status check_cache(const crc_cache* c, const crc_shape* sh) {
  if (!c || !c->k.data || !c->v.data) return CRC_ERR_INVALID_ARG;
  if (c->n_keys < 1 || c->nseg < 0 || c->nseg > CRC_MAX_SEGMENTS) return CRC_ERR_SHAPE;
  if (c->k.stride_head != sh->d || c->k.stride_token < (int64_t)sh->H * sh->d ||
      c->k.stride_layer < (int64_t)c->n_keys * c->k.stride_token)
    return CRC_ERR_SHAPE;
  if (c->v.stride_head != c->k.stride_head || c->v.stride_token != c->k.stride_token ||
      c->v.stride_layer != c->k.stride_layer)
    return CRC_ERR_SHAPE;
  const int es = elem_bytes(sh->dtype);
  if (!aligned16(c->k.data) || !aligned16(c->v.data) || (c->k.stride_token * es) % 16 != 0 ||
      (c->k.stride_layer * es) % 16 != 0 || ((int64_t)sh->H * sh->d * es) % 16 != 0)
    return CRC_ERR_UNSUPPORTED;
  const int32_t nc = sh->F * sh->h * sh->w;
  for (int g = 0; g < c->nseg; ++g) {
    const crc_segment& s = c->seg[g];
    if (s.offset < 0 || s.length < 0 || (int64_t)s.offset + s.length > c->n_keys) return CRC_ERR_SHAPE;
    if (s.kind != CRC_SEG_SINK && s.kind != CRC_SEG_RETRIEVED && s.kind != CRC_SEG_WINDOW && s.kind != CRC_SEG_CURRENT)
      return CRC_ERR_INVALID_ARG;
    if (s.kind == CRC_SEG_RETRIEVED && (s.slot < 0 || s.slot >= CRC_MAX_K || (s.length != 0 && s.length != nc)))
      return CRC_ERR_SHAPE;
    if (s.kind == CRC_SEG_CURRENT && s.length != 0 && s.length != nc) return CRC_ERR_SHAPE;
    for (int h2 = 0; h2 < g; ++h2) {  // segments may not overlap
      const crc_segment& o = c->seg[h2];
      if (s.length > 0 && o.length > 0 && s.offset < o.offset + o.length && o.offset < s.offset + s.length)
        return CRC_ERR_SHAPE;
    }
  }
  return CRC_OK;
}

// RoPE layout limits of crc_rope (see include/crc.h).
crc_status check_rope(const crc_rope* r, const crc_shape* sh) {
  if (!r || r->pairs == 0) return CRC_OK;
  if (r->pairs < 0 || r->pairs > CRC_MAX_ROPE_PAIRS || r->channel0 < 0 || !(r->theta > 0.0) || !isfinite(r->theta) ||
      (r->interleaved != 0 && r->interleaved != 1))
    return CRC_ERR_INVALID_ARG;
  if ((int64_t)r->channel0 + 2LL * r->pairs > sh->d) return CRC_ERR_INVALID_ARG;
  const int epv = 16 / elem_bytes(sh->dtype);  // elements per 16-byte vector
  if (r->interleaved ? (r->channel0 % 2 != 0) : (r->channel0 % epv != 0 || r->pairs % epv != 0))
    return CRC_ERR_UNSUPPORTED;
  return CRC_OK;
}

// Gather arguments for the retrieved segments of `cache` from a slab pool.
crc_status fill_gather(crc::GatherArgs& g, const crc_shape* sh, const void* pool, int32_t num_slabs,
                       const crc_cache* cache, int32_t k, const crc_rope* rope) {
  crc_status st = check_cache(cache, sh);
  if (st) return st;
  if ((st = check_rope(rope, sh))) return st;
  if (!pool || num_slabs < 1) return CRC_ERR_INVALID_ARG;
  if (!aligned16(pool)) return CRC_ERR_UNSUPPORTED;
  const int es = elem_bytes(sh->dtype);
  const int32_t nc = sh->F * sh->h * sh->w;
  const int32_t row_bytes = sh->H * sh->d * es;
  g.pool = static_cast<const char*>(pool);
  g.num_slabs = num_slabs;
  g.kv_bytes = (int64_t)sh->L * nc * row_bytes;
  g.slab_bytes = 2 * g.kv_bytes;
  g.cache_k = static_cast<char*>(cache->k.data);
  g.cache_v = static_cast<char*>(cache->v.data);
  g.cache_layer_stride = cache->k.stride_layer * es;
  g.cache_token_stride = cache->k.stride_token * es;
  g.L = sh->L;
  g.Nc = nc;
  g.row_bytes = row_bytes;
  g.d = sh->d;
  g.elem_bytes = es;
  g.F = sh->F;
  for (int r = 0; r < CRC_MAX_K; ++r) g.slot_offset[r] = -1;
  for (int i = 0; i < cache->nseg; ++i) {
    const crc_segment& sg = cache->seg[i];
    if (sg.kind == CRC_SEG_RETRIEVED && sg.slot < k && sg.length == nc) {
      if (g.slot_offset[sg.slot] >= 0) return CRC_ERR_SHAPE;  // two segments for one slot
      g.slot_offset[sg.slot] = sg.offset;
    }
  }
  g.rope_pairs = 0;
  if (rope && rope->pairs > 0) {
    g.rope_pairs = rope->pairs;
    g.rope_c0 = rope->channel0;
    g.rope_interleaved = rope->interleaved;
    g.rope_pos_slot0 = rope->pos_slot0;
    g.rope_pos_stride = rope->pos_stride;
    g.rope_frame_pos0 = rope->frame_pos0;
    for (int i = 0; i < rope->pairs; ++i) g.rope_omega[i] = pow(rope->theta, -((double)i / (double)rope->pairs));
  }
  return CRC_OK;
}

void pack_frames(crc::FrameSet& fs, const crc_frame* fr, int F) {
  memset(&fs, 0, sizeof(fs));
  fs.F = F;
  for (int f = 0; f < F; ++f) {
    memcpy(&fs.rec[f][0], fr[f].K, 9 * sizeof(double));
    memcpy(&fs.rec[f][9], fr[f].R, 9 * sizeof(double));
    memcpy(&fs.rec[f][18], fr[f].c, 3 * sizeof(double));
  }
}

// ---- validation and argument set-up of each entry point -----------------------
// Each prep_* checks every argument of its call on the host and fills the launch
// arguments; nothing is enqueued.  A null `frames` / `cur` means the per-step values
// come from a crc_step descriptor on the device (crc_chunk_step).

crc_status prep_cache_update(crc::CacheUpdateArgs& a, const crc_bank* bank, const crc_shape* shape, int32_t chunk,
                             const crc_frame* frames, const float* d_depth, const void* d_k, const void* d_v,
                             const crc_cache* cache, int32_t window_offset) {
  crc_status st = check_shape(shape);
  if (st) return st;
  const bool with_kv = d_k != nullptr || d_v != nullptr;
  if ((st = check_bank(bank, with_kv))) return st;
  if (!d_depth || chunk < 0 || chunk >= bank->capacity) return CRC_ERR_INVALID_ARG;
  if ((d_k == nullptr) != (d_v == nullptr)) return CRC_ERR_INVALID_ARG;
  if (frames && !frames_ok(frames, shape->F)) return CRC_ERR_INVALID_ARG;
  const int es = elem_bytes(shape->dtype);
  const int32_t nc = shape->F * shape->h * shape->w;
  const int32_t row_bytes = shape->H * shape->d * es;
  if (with_kv && (!aligned16(d_k) || !aligned16(d_v) || !aligned16(bank->kv) || row_bytes % 16 != 0))
    return CRC_ERR_UNSUPPORTED;
  memset(&a, 0, sizeof(a));
  if (frames) pack_frames(a.frames, frames, shape->F);
  a.frames.F = shape->F;
  a.capacity = bank->capacity;
  a.num_slabs = bank->num_slabs;
  a.depth_base = bank->depth;
  a.slab_chunk = bank->slab_chunk;
  a.bank_frames = bank->frames;
  a.bank_centre = bank->centre;
  a.bank_view = bank->view;
  a.chunk = chunk;
  a.depth_src = d_depth;
  a.depth_count = nc;
  a.depth_dst = bank->depth + (int64_t)chunk * nc;
  a.L = shape->L;
  a.Nc = nc;
  a.row_bytes = row_bytes;
  if (with_kv) {
    a.k_src = static_cast<const char*>(d_k);
    a.v_src = static_cast<const char*>(d_v);
    a.slab_bytes = 2LL * shape->L * nc * row_bytes;
    a.kv_base = static_cast<char*>(bank->kv);
    a.slab = a.kv_base + (int64_t)(chunk % bank->num_slabs) * a.slab_bytes;
    a.slab_owner = bank->slab_chunk ? bank->slab_chunk + chunk % bank->num_slabs : nullptr;
    if (window_offset >= 0) {
      if ((st = check_cache(cache, shape))) return st;
      if ((int64_t)window_offset + nc > cache->n_keys) return CRC_ERR_SHAPE;
      a.cache_k = static_cast<char*>(cache->k.data);
      a.cache_v = static_cast<char*>(cache->v.data);
      a.n_keys = cache->n_keys;
      a.win_k = a.cache_k + (int64_t)window_offset * cache->k.stride_token * es;
      a.win_v = a.cache_v + (int64_t)window_offset * cache->v.stride_token * es;
      a.win_layer_stride = cache->k.stride_layer * es;
      a.win_token_stride = cache->k.stride_token * es;
    }
  }
  return CRC_OK;
}

crc_status prep_retrieve(crc::RetrieveArgs& a, crc::GatherArgs& g, const crc_bank* bank, int32_t bank_count,
                         const crc_shape* shape, const crc_frame* cur, int32_t n, const crc_retrieval* p,
                         const crc_cache* cache, const crc_rope* rope, int32_t* d_idx, double* d_score,
                         int32_t* d_count, void* d_workspace, size_t workspace_bytes) {
  crc_status st = check_shape(shape);
  if (st) return st;
  if ((st = check_bank(bank, cache != nullptr))) return st;
  if (!p || !d_idx || !d_count) return CRC_ERR_INVALID_ARG;
  if (bank_count < 0 || bank_count > bank->capacity || n < 0) return CRC_ERR_INVALID_ARG;
  if (p->k < 1 || p->k > CRC_MAX_K || !(p->E > 0.0) || !isfinite(p->E) || !isfinite(p->w_v) || isnan(p->tau_c) ||
      isnan(p->cos_tau_v) || p->ext_min < 0)
    return CRC_ERR_INVALID_ARG;
  if (cur && !frames_ok(cur, shape->F)) return CRC_ERR_INVALID_ARG;
  const size_t ws = crc::retrieve_workspace_bytes(bank_count, p->k);
  if (ws > 0 && (!d_workspace || workspace_bytes < ws || !aligned16(d_workspace))) return CRC_ERR_INVALID_ARG;
  if ((st = check_rope(rope, shape))) return st;
  memset(&a, 0, sizeof(a));
  if (cur) pack_frames(a.cur, cur, shape->F);
  a.cur.F = shape->F;
  a.capacity = bank->capacity;
  a.centre = bank->centre;
  a.view = bank->view;
  a.slab_chunk = bank->slab_chunk;
  a.num_slabs = bank->num_slabs;
  if (ws > 0) {
    a.partial = static_cast<crc::TopkCand*>(d_workspace);
    a.ticket = reinterpret_cast<unsigned int*>(static_cast<char*>(d_workspace) + ws - 256);
  }
  a.count = bank_count;
  a.n = n;
  a.E = p->E;
  a.w_v = p->w_v;
  a.tau_c = p->tau_c;
  a.cos_tau_v = p->cos_tau_v;
  a.delta = p->delta;
  a.k = p->k;
  a.ext_first = p->ext_first;
  a.ext_min = p->ext_min;
  a.exclude_sink = p->exclude_sink != 0;
  a.d_idx = d_idx;
  a.d_score = d_score;
  a.d_count = d_count;
  memset(&g, 0, sizeof(g));
  g.pool = nullptr;
  if (cache && (st = fill_gather(g, shape, bank->kv, bank->num_slabs, cache, p->k, rope))) return st;
  return CRC_OK;
}

crc_status prep_correspond(crc::CorrespondArgs& a, const crc_shape* shape, const crc_frame* cur, const float* d_depth,
                           const crc_bank* bank, const int32_t* d_idx, const int32_t* d_count, int32_t k, float eps,
                           float* d_uv, int32_t* d_cell, uint8_t* d_valid) {
  crc_status st = check_shape(shape);
  if (st) return st;
  if ((st = check_bank(bank, false))) return st;
  if (!d_depth || !d_idx || !d_uv || !d_valid) return CRC_ERR_INVALID_ARG;
  if (k < 1 || k > CRC_MAX_K || isnan(eps) || eps < 0.f) return CRC_ERR_INVALID_ARG;
  if (cur && !frames_ok(cur, shape->F)) return CRC_ERR_INVALID_ARG;
  if (((uintptr_t)d_uv & 7u) != 0) return CRC_ERR_UNSUPPORTED;
  // the kernel addresses the bank's depth array with 32-bit offsets
  if ((int64_t)bank->capacity * shape->F * shape->h * shape->w > INT32_MAX) return CRC_ERR_UNSUPPORTED;
  memset(&a, 0, sizeof(a));
  if (cur) pack_frames(a.cur, cur, shape->F);
  a.cur.F = shape->F;
  a.depth = d_depth;
  a.bank_frames = bank->frames;
  a.bank_depth = bank->depth;
  a.capacity = bank->capacity;
  a.d_idx = d_idx;
  a.d_count = d_count;
  a.k = k;
  a.F = shape->F;
  a.h = shape->h;
  a.w = shape->w;
  a.eps = eps;
  a.uv = d_uv;
  a.cell = d_cell;
  a.valid = d_valid;
  return CRC_OK;
}

// `tc` is set when the call runs on the tensor-core kernel.
crc_status prep_attention(crc::AttnArgs& a, bool& tc, const crc_shape* shape, crc_tensor q, const crc_cache* cache,
                          crc_tensor o, float* d_lse, int32_t n_q, const float* d_uv, const uint8_t* d_valid, int32_t k,
                          const int32_t* d_slot_chunk, float lambda, float sigma, int32_t flags, int32_t* d_status) {
  crc_status st = check_shape(shape);
  if (st) return st;
  if ((st = check_cache(cache, shape))) return st;
  if (!q.data || !o.data) return CRC_ERR_INVALID_ARG;
  const int32_t nc = shape->F * shape->h * shape->w;
  if (n_q != nc) return CRC_ERR_SHAPE;
  if (k < 0 || k > CRC_MAX_K || !isfinite(lambda) || lambda < 0.f || !(sigma > 0.f) || !isfinite(sigma))
    return CRC_ERR_INVALID_ARG;
  if (flags & ~(CRC_ATTN_SIMT | CRC_ATTN_GAUSSIAN | CRC_ATTN_SKIP_FAR | CRC_ATTN_BIAS_DIRECT | CRC_ATTN_FRAME_CAUSAL))
    return CRC_ERR_INVALID_ARG;
  bool any_ret = false, any_other = false;
  for (int g = 0; g < cache->nseg; ++g) {
    if (cache->seg[g].kind == CRC_SEG_RETRIEVED && cache->seg[g].length > 0) {
      any_ret = true;
      if (cache->seg[g].slot >= k) return CRC_ERR_SHAPE;
    } else if (cache->seg[g].length > 0) {
      any_other = true;
    }
  }
  if (any_ret && (!d_uv || !d_valid)) return CRC_ERR_INVALID_ARG;
  // the kernels read each correspondence as one float2
  if (((uintptr_t)d_uv & 7u) != 0) return CRC_ERR_UNSUPPORTED;
  if (q.stride_head < shape->d || q.stride_token < (int64_t)shape->H * q.stride_head ||
      o.stride_head < shape->d || o.stride_token < (int64_t)shape->H * o.stride_head)
    return CRC_ERR_SHAPE;
  memset(&a, 0, sizeof(a));
  a.q = q.data;
  a.k = cache->k.data;
  a.v = cache->v.data;
  a.o = o.data;
  a.lse = d_lse;
  a.q_sl = q.stride_layer;
  a.q_st = q.stride_token;
  a.q_sh = q.stride_head;
  a.k_sl = cache->k.stride_layer;
  a.k_st = cache->k.stride_token;
  a.k_sh = cache->k.stride_head;
  a.o_sl = o.stride_layer;
  a.o_st = o.stride_token;
  a.o_sh = o.stride_head;
  a.L = shape->L;
  a.H = shape->H;
  a.d = shape->d;
  a.Nq = n_q;
  a.Nk = cache->n_keys;
  a.F = shape->F;
  a.h = shape->h;
  a.w = shape->w;
  a.S = k * shape->F;
  a.nseg = cache->nseg;
  for (int g = 0; g < cache->nseg; ++g) a.seg[g] = cache->seg[g];
  a.uv = d_uv;
  a.valid = d_valid;
  a.slot_chunk = d_slot_chunk;
  a.lambda = lambda;
  a.sigma = sigma;
  a.dtype = shape->dtype;
  a.status = d_status;
  a.bias_form = (flags & CRC_ATTN_GAUSSIAN) ? 1 : 0;
  a.bias_direct = (flags & CRC_ATTN_BIAS_DIRECT) ? 1 : 0;
  a.frame_causal = (flags & CRC_ATTN_FRAME_CAUSAL) ? 1 : 0;
  // skipped weights are scaled by at most 2^-64: lambda d^2 / (2 sigma^2) >= 64 ln 2
  a.skip_far = (flags & CRC_ATTN_SKIP_FAR) && !(flags & CRC_ATTN_GAUSSIAN) && lambda > 0.f && any_ret && any_other &&
                       d_valid
                   ? 1
                   : 0;
  a.skip_d2 = lambda > 0.f ? (float)(2.0 * (double)sigma * (double)sigma * 64.0 * 0.6931471805599453 / (double)lambda)
                           : INFINITY;
  tc = shape->dtype == CRC_BF16 && !(flags & CRC_ATTN_SIMT);
  if (!(tc ? crc::attn_tc_supported(a) : crc::attn_simt_supported(a))) return CRC_ERR_UNSUPPORTED;
  return CRC_OK;
}

}  // namespace

extern "C" {

const char* crc_version(void) { return "crc 0.1.0 (sm_103a)"; }

const char* crc_status_string(crc_status st) {
  switch (st) {
    case CRC_OK: return "ok";
    case CRC_ERR_INVALID_ARG: return "invalid argument";
    case CRC_ERR_SHAPE: return "inconsistent shape or stride";
    case CRC_ERR_UNSUPPORTED: return "unsupported dtype, head dim, alignment or device";
    case CRC_ERR_CUDA: return "CUDA error";
    case CRC_ERR_DEVICE: return "kernel reported a failure";
    case CRC_ERR_TOO_LARGE: return "beyond the fixed scratch of the no-allocation entry point";
    default: return "unknown status";
  }
}

int32_t crc_last_cuda_error(void) { return g_last_cuda_error; }

crc_status crc_bank_insert_poses(const crc_bank* bank, const crc_shape* shape, int32_t first, int32_t count,
                                 const crc_frame* frames, cudaStream_t s) {
  CRC_RANGE("crc_bank_insert_poses");
  crc_status st = check_shape(shape);
  if (st) return st;
  if ((st = check_bank(bank, false))) return st;
  if (count < 0 || first < 0 || (count > 0 && !frames)) return CRC_ERR_INVALID_ARG;
  if ((int64_t)first + count > bank->capacity) return CRC_ERR_INVALID_ARG;
  if (count == 0) return CRC_OK;
  for (int32_t j = 0; j < count; ++j)
    if (!frames_ok(frames + (int64_t)j * shape->F, shape->F)) return CRC_ERR_INVALID_ARG;
  // crc_frame is exactly 21 packed doubles, the record layout of the bank
  static_assert(sizeof(crc_frame) == crc::kFrameDoubles * sizeof(double), "crc_frame layout");
  cudaError_t e = cudaMemcpyAsync(bank->frames + (int64_t)first * shape->F * crc::kFrameDoubles, frames,
                                  (size_t)count * shape->F * sizeof(crc_frame), cudaMemcpyHostToDevice, s);
  if (e != cudaSuccess) return cuda_fail(e);
  crc::PoseInsertArgs a{bank->frames, bank->centre, bank->view, shape->F, first, count};
  e = crc::launch_pose_summary(a, s);
  return e == cudaSuccess ? CRC_OK : cuda_fail(e);
}

crc_status crc_cache_update(const crc_bank* bank, const crc_shape* shape, int32_t chunk, const crc_frame* frames,
                            const float* d_depth, const void* d_k, const void* d_v, const crc_cache* cache,
                            int32_t window_offset, cudaStream_t s) {
  CRC_RANGE("crc_cache_update");
  crc::CacheUpdateArgs a;
  crc_status st = prep_cache_update(a, bank, shape, chunk, frames, d_depth, d_k, d_v, cache, window_offset);
  if (st) return st;
  cudaError_t e = crc::launch_cache_update(a, s);
  return e == cudaSuccess ? CRC_OK : cuda_fail(e);
}

size_t crc_retrieve_workspace_size(int32_t bank_count, int32_t k) {
  if (bank_count < 0 || k < 1 || k > CRC_MAX_K) return 0;
  return crc::retrieve_workspace_bytes(bank_count, k);
}

crc_status crc_retrieve(const crc_bank* bank, int32_t bank_count, const crc_shape* shape, const crc_frame* cur,
                        int32_t n, const crc_retrieval* p, const crc_cache* cache, const crc_rope* rope,
                        int32_t* d_idx, double* d_score, int32_t* d_count, void* d_workspace, size_t workspace_bytes,
                        cudaStream_t s) {
  CRC_RANGE("crc_retrieve");
  crc::RetrieveArgs a;
  crc::GatherArgs g;
  crc_status st = prep_retrieve(a, g, bank, bank_count, shape, cur, n, p, cache, rope, d_idx, d_score, d_count,
                                d_workspace, workspace_bytes);
  if (st) return st;
  cudaError_t e = crc::launch_retrieve(a, g, s);
  return e == cudaSuccess ? CRC_OK : cuda_fail(e);
}

crc_status crc_gather(const crc_shape* shape, const void* pool, int32_t num_slabs, const int32_t* d_idx, int32_t k,
                      const crc_cache* cache, const crc_rope* rope, cudaStream_t s) {
  CRC_RANGE("crc_gather");
  crc_status st = check_shape(shape);
  if (st) return st;
  if (!d_idx || !cache || k < 1 || k > CRC_MAX_K) return CRC_ERR_INVALID_ARG;
  crc::GatherOnlyArgs a;
  memset(&a, 0, sizeof(a));
  a.d_idx = d_idx;
  a.k = k;
  if ((st = fill_gather(a.g, shape, pool, num_slabs, cache, k, rope))) return st;
  cudaError_t e = crc::launch_gather(a, s);
  return e == cudaSuccess ? CRC_OK : cuda_fail(e);
}

crc_status crc_correspond(const crc_shape* shape, const crc_frame* cur, const float* d_depth, const crc_bank* bank,
                          const int32_t* d_idx, const int32_t* d_count, int32_t k, float eps, float* d_uv,
                          int32_t* d_cell, uint8_t* d_valid, cudaStream_t s) {
  CRC_RANGE("crc_correspond");
  crc::CorrespondArgs a;
  crc_status st = prep_correspond(a, shape, cur, d_depth, bank, d_idx, d_count, k, eps, d_uv, d_cell, d_valid);
  if (st) return st;
  cudaError_t e = crc::launch_correspond(a, s);
  return e == cudaSuccess ? CRC_OK : cuda_fail(e);
}

crc_status crc_biased_attention(const crc_shape* shape, crc_tensor q, const crc_cache* cache, crc_tensor o,
                                float* d_lse, int32_t n_q, const float* d_uv, const uint8_t* d_valid, int32_t k,
                                const int32_t* d_slot_chunk, float lambda, float sigma, int32_t flags,
                                int32_t* d_status, cudaStream_t s) {
  CRC_RANGE("crc_biased_attention");
  crc::AttnArgs a;
  bool tc = false;
  crc_status st = prep_attention(a, tc, shape, q, cache, o, d_lse, n_q, d_uv, d_valid, k, d_slot_chunk, lambda, sigma,
                                 flags, d_status);
  if (st) return st;
  cudaError_t e = tc ? crc::launch_attn_tc(a, s) : crc::launch_attn_simt(a, s);
  return e == cudaSuccess ? CRC_OK : cuda_fail(e);
}

crc_status crc_chunk_step(const crc_step_plan* plan, const crc_step* d_step, cudaStream_t s) {
  CRC_RANGE("crc_chunk_step");
  if (!plan || !d_step || ((uintptr_t)d_step & 7u) != 0 || !plan->d_status) return CRC_ERR_INVALID_ARG;
  const crc_shape* shape = &plan->shape;
  const crc_bank* bank = &plan->bank;
  const crc_cache* cache = &plan->cache;
  const int32_t nc = shape->F * shape->h * shape->w;
  // every check of the four calls, before anything is enqueued; the per-step values are
  // placeholders here (chunk 0, window slot 0, all bank entries) and come from the descriptor
  crc::CacheUpdateArgs cu;
  crc_status st = prep_cache_update(cu, bank, shape, 0, nullptr, plan->d_depth, plan->d_k, plan->d_v, cache, 0);
  if (st) return st;
  if (!plan->d_k) return CRC_ERR_INVALID_ARG;
  crc::RetrieveArgs ra;
  crc::GatherArgs g;
  const crc_rope* rope = plan->rope.pairs > 0 ? &plan->rope : nullptr;
  if ((st = prep_retrieve(ra, g, bank, bank->capacity, shape, nullptr, 0, &plan->retrieval, cache, rope, plan->d_idx,
                          plan->d_score, plan->d_count, plan->d_workspace, plan->workspace_bytes)))
    return st;
  crc::CorrespondArgs ca;
  if ((st = prep_correspond(ca, shape, nullptr, plan->d_depth, bank, plan->d_idx, plan->d_count, plan->retrieval.k,
                            plan->eps, plan->d_uv, plan->d_cell, plan->d_valid)))
    return st;
  crc::AttnArgs aa;
  bool tc = false;
  if ((st = prep_attention(aa, tc, shape, plan->q, cache, plan->o, plan->d_lse, nc, plan->d_uv, plan->d_valid,
                           plan->retrieval.k, plan->d_idx, plan->lambda, plan->sigma, plan->attn_flags,
                           plan->d_status)))
    return st;
  cu.step = ra.step = g.step = ca.step = aa.step = d_step;
  cu.status = ra.status = plan->d_status;
  cudaError_t e = crc::launch_cache_update(cu, s);
  if (e == cudaSuccess) e = crc::launch_retrieve(ra, g, s);
  if (e == cudaSuccess) e = crc::launch_correspond(ca, s);
  if (e == cudaSuccess) e = tc ? crc::launch_attn_tc(aa, s) : crc::launch_attn_simt(aa, s);
  return e == cudaSuccess ? CRC_OK : cuda_fail(e);
}

double crc_bias_expansion_bound(float lambda, float sigma, int32_t h, int32_t w) {
  return crc::bias_expansion_bound(lambda, sigma, h, w);
}

}  // extern "C"

namespace crc {
crc_status record_cuda_error(cudaError_t e) { return cuda_fail(e); }
}  // namespace crc
