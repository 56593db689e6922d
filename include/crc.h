/*
 * crc.h — C ABI of the per-chunk revisit-consistency attention path.
 *
 * The path implements the inference-time method of "Closing the Loop:
 * Training-Free Revisit Consistency for Autoregressive Generative Rendering":
 *
 *   crc_cache_update      Sec. 4.2  "Cache layout": the new chunk enters the recent
 *                                   window; its K/V, depth and poses are retained
 *                                   outside the attention cache (the memory bank).
 *   crc_retrieve          Sec. 4.2, Eq. 1: score every historical chunk against the
 *                                   current chunk's pose, gate, take the top-k, and
 *                                   gather their K/V into the retrieved cache slots;
 *                                   an empty admissible set extends the recent window.
 *   crc_correspond        Sec. 4.3, Eq. 3-4: reproject each query token through its
 *                                   depth and the relative pose into every retrieved
 *                                   frame; visibility test; exact-fallback flags.
 *   crc_biased_attention  Sec. 4.3, Eq. 2: softmax(q.k/sqrt(d) + lambda B) V, with the
 *                                   Gaussian correspondence bias B computed inside the
 *                                   tile loop on retrieved key columns only.
 *
 * Conventions shared by every entry point:
 *   - All device pointers are caller-owned.  No entry point allocates or frees
 *     memory; none keeps state between calls.
 *   - Work is enqueued on the caller's stream `s`; results are valid once the
 *     caller synchronises that stream.  No entry point synchronises the host,
 *     except that host arrays passed by pointer are read before the call returns.
 *   - Every argument is validated on the host before anything is enqueued; a
 *     failed check returns an error code and enqueues nothing.
 *   - Tensors of attention data use the token-major layout [L][N][H][d]
 *     (layer, token, head, head-dim) with d contiguous; strides are in elements.
 *   - Grid coordinates: token (row i, col j) of an h x w frame is the point
 *     (x, y) = (j, i); tokens of a chunk are ordered frame, row, col.
 */
#ifndef CRC_H_
#define CRC_H_

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes -------------------------------------------------------- */
typedef int32_t crc_status;
#define CRC_OK 0
#define CRC_ERR_INVALID_ARG 1  /* null pointer, negative size, bad parameter value */
#define CRC_ERR_SHAPE 2        /* inconsistent sizes or strides                   */
#define CRC_ERR_UNSUPPORTED 3  /* dtype / head dim / alignment / device not handled */
#define CRC_ERR_CUDA 4         /* a CUDA call failed; see crc_last_cuda_error()     */
#define CRC_ERR_DEVICE 5       /* a kernel reported a failure in its status word    */
#define CRC_ERR_TOO_LARGE 6    /* beyond the fixed scratch of crc_retrieve_noalloc  */

/* ---- element types ------------------------------------------------------- */
#define CRC_F32 0
#define CRC_BF16 1

/* ---- cache segment kinds (Sec. 4.2 "Cache layout") ----------------------- */
#define CRC_SEG_SINK 0       /* the anchor: the first chunk, never evicted          */
#define CRC_SEG_RETRIEVED 1  /* a pose-retrieved slot; `slot` = retrieval rank r    */
#define CRC_SEG_WINDOW 2     /* the recent window (including the current chunk)     */
#define CRC_SEG_CURRENT 3    /* the window slot holding the current chunk (length N_c or 0): a
                                window segment, except under CRC_ATTN_FRAME_CAUSAL     */

#define CRC_MAX_SEGMENTS 16
#define CRC_MAX_FRAMES 4   /* frames per chunk, F */
#define CRC_MAX_K 8        /* retrieved slots per step, k */
#define CRC_MAX_ROPE_PAIRS 64  /* temporal rotary pairs per head, crc_rope.pairs */

/* One latent frame's camera annotation (Sec. 4.1): intrinsics K rescaled to the
 * token grid, camera-to-world rotation R and camera centre c, all row-major fp64.
 * K must have last row (0, 0, 1). */
typedef struct {
  double K[9];
  double R[9];
  double c[3];
} crc_frame;

/* Problem shape of one call. */
typedef struct {
  int32_t L;      /* layers handled by the call                         */
  int32_t H;      /* attention heads                                    */
  int32_t d;      /* head dimension (64 or 128)                         */
  int32_t F;      /* latent frames per chunk (1..CRC_MAX_FRAMES)         */
  int32_t h, w;   /* token grid of one latent frame; N_c = F*h*w tokens */
  int32_t dtype;  /* CRC_F32 or CRC_BF16                                 */
} crc_shape;

/* A [L][N][H][d] tensor: element (l, n, hd, e) is at
 * data[l*stride_layer + n*stride_token + hd*stride_head + e]. */
typedef struct {
  void* data;
  int64_t stride_layer;
  int64_t stride_token;
  int64_t stride_head;
} crc_tensor;

/* Contiguous key range [offset, offset+length) of the cache.  Keys outside every
 * segment are masked.  A zero-length segment is allowed and contributes nothing. */
typedef struct {
  int32_t offset;
  int32_t length;
  int32_t kind;  /* CRC_SEG_* */
  int32_t slot;  /* retrieval rank r for CRC_SEG_RETRIEVED (length must be N_c) */
} crc_segment;

/* The segmented clean KV cache [sink | retrieved slots | recent window]. */
typedef struct {
  crc_tensor k;  /* [L][n_keys][H][d]                                      */
  crc_tensor v;  /* same layout and strides as k                           */
  int32_t n_keys;
  int32_t nseg;
  crc_segment seg[CRC_MAX_SEGMENTS];
} crc_cache;

/* Memory bank of the chunks generated so far (Sec. 4.2: chunks evicted from the
 * recent window stay retrievable).  Device arrays, caller-allocated:
 *   frames [capacity][F][21]  fp64 crc_frame records of every chunk
 *   centre [capacity][3]      fp64 chunk centre c_j (written by the library)
 *   view   [capacity][3]      fp64 unit view direction v_j (written by the library)
 *   depth  [capacity][F][h][w] fp32 planar metric depth of every chunk
 *   kv     [num_slabs][2][L][N_c][H][d] K (index 0) and V (index 1) slabs, dense,
 *          dtype of the call; chunk j lives in slab j % num_slabs.
 *   slab_chunk [num_slabs] int32, or NULL: the chunk whose K/V slab s holds (-1 for
 *          none; the caller fills it with -1 before the first update).  When it is
 *          given, crc_cache_update records every chunk it writes, and retrieval only
 *          admits chunks whose slab still holds them: with num_slabs < capacity a
 *          chunk stops being retrievable once chunk j + num_slabs overwrites its slab.
 *          When it is NULL the caller guarantees that slab j % num_slabs holds chunk
 *          j's K/V for every chunk that can be retrieved (e.g. num_slabs >= the
 *          number of chunks, or a pool of synthetic slabs).
 * Poses, pose summaries and depth are kept for all `capacity` chunks. */
typedef struct {
  int32_t capacity;
  int32_t num_slabs;
  double* frames;
  double* centre;
  double* view;
  float* depth;
  void* kv;
  int32_t* slab_chunk;
} crc_bank;

/* Eq. 1 parameters and the empty-set fallback of Sec. 4.2. */
typedef struct {
  double E;          /* scene-scale normaliser of the distance term (> 0)          */
  double w_v;        /* weight of the angular term (0.5 in the paper)              */
  double tau_c;      /* distance gate on ||c_j - c_n|| / E (may be +inf)           */
  double cos_tau_v;  /* angle gate: admissible iff v_j . v_n >= cos_tau_v          */
  int32_t delta;     /* temporal gap: admissible iff n - j >= delta                */
  int32_t k;         /* retrieved slots (1..CRC_MAX_K)                             */
  int32_t ext_first; /* fallback: slot r >= count holds chunk ext_first-(r-count)  */
  int32_t ext_min;   /*   if that is >= ext_min (else the slot stays empty);       */
                     /*   ext_first < 0 disables the fallback                      */
  int32_t exclude_sink; /* non-zero: chunk 0 (the anchor, always cached) is never  */
                        /*   admissible; 0 keeps the literal reading of Eq. 1      */
} crc_retrieval;

/* RoPE re-positioning of re-packed chunks (Sec. 4.2 "Cache packing": a retrieved
 * chunk is re-packed at rotary positions adjacent to the recent window).
 *
 * Keys are cached after their rotary embedding, at the temporal position of the
 * latent frame that produced them: frame f of chunk j sits at
 * frame_pos0 + j*F + f.  Gathered into retrieved slot r, that frame is moved to
 * pos_slot0 + r*pos_stride + f, i.e. every temporal rotary pair i of every head is
 * multiplied, as the complex number k[a] + i k[b], by exp(i delta_r omega_i) with
 *   omega_i = theta^(-i / pairs),  delta_r = pos_slot0 + r*pos_stride - frame_pos0 - j*F.
 * Pair i occupies channels (channel0 + 2i, channel0 + 2i + 1) of the head when
 * `interleaved`, else (channel0 + i, channel0 + i + pairs).  Only the temporal
 * block is rotated (the spatial rotary axes of a chunk do not move) and values
 * carry no rotary embedding.  The rotation runs in fp32 with fp64 angles and is
 * rounded once to the cache dtype.  pairs = 0 (or a NULL crc_rope) copies the
 * keys unchanged.  Layout limits: channel0 + 2*pairs <= d, pairs <= 64; with
 * `interleaved` channel0 is even; without it channel0 and pairs are multiples of
 * 16 bytes' worth of elements (8 for bf16, 4 for fp32). */
typedef struct {
  int32_t channel0;
  int32_t pairs;
  int32_t interleaved;
  int32_t pos_slot0;
  int32_t pos_stride;
  int32_t frame_pos0;
  double theta;
} crc_rope;

/* ---- library information ------------------------------------------------- */
const char* crc_version(void);
const char* crc_status_string(crc_status st);
/* The cudaError_t of the last CRC_ERR_CUDA returned on this thread. */
int32_t crc_last_cuda_error(void);

/*
 * crc_bank_insert_poses — record the camera annotations of chunks
 * [first, first+count) in the bank and compute each chunk's centre and view
 * direction (Sec. 4.2, the (c_j, v_j) of Eq. 1).
 *
 *   frames  host array [count][F] of crc_frame; copied to bank->frames.
 * The chunk centre is the mean of its frames' centres and the view direction is
 * the normalised sum of their optical axes (third column of R), in frame order,
 * computed in fp64 without fused multiply-add.
 * Errors: CRC_ERR_INVALID_ARG (null pointers, count < 0, first+count > capacity).
 */
crc_status crc_bank_insert_poses(const crc_bank* bank, const crc_shape* shape, int32_t first, int32_t count,
                                 const crc_frame* frames, cudaStream_t s);

/*
 * crc_cache_update — Sec. 4.2 "Cache layout": chunk `chunk` (its K/V just
 * produced by the clean-context pass) enters the recent window and the bank.
 *
 *   frames       host [F] crc_frame of the chunk; stored in the bank with its
 *                centre and view direction (as crc_bank_insert_poses).
 *   d_depth      device [F][h][w] fp32 depth; copied to bank->depth[chunk].
 *   d_k, d_v     device [L][N_c][H][d] dense, dtype of the call; copied to slab
 *                chunk % num_slabs of bank->kv (and bank->slab_chunk[chunk %
 *                num_slabs] = chunk when the bank tracks its slabs) and, if
 *                window_offset >= 0, to cache keys [window_offset, window_offset + N_c)
 *                of every layer.  Both may be NULL (poses and depth only).
 *   cache        may be NULL when window_offset < 0.
 * The sink and the other cache keys are not touched.
 * Errors: CRC_ERR_INVALID_ARG, CRC_ERR_SHAPE (window slot outside the cache),
 * CRC_ERR_UNSUPPORTED (cache not dense per token), CRC_ERR_CUDA.
 */
crc_status crc_cache_update(const crc_bank* bank, const crc_shape* shape, int32_t chunk, const crc_frame* frames,
                            const float* d_depth, const void* d_k, const void* d_v, const crc_cache* cache,
                            int32_t window_offset, cudaStream_t s);

/*
 * crc_retrieve — Sec. 4.2, Eq. 1 over bank chunks j in [0, bank_count):
 *   s(j) = ||c_j - c_n||_2 / E + w_v (1 - v_j . v_n)
 *   A_n  = { j : ||c_j - c_n||/E <= tau_c, v_j . v_n >= cos_tau_v, n - j >= delta }
 * restricted, when bank->slab_chunk is given, to chunks whose K/V slab still holds
 * them (a window-extension chunk whose slab was overwritten leaves its slot empty)
 * where (c_n, v_n) summarise `cur` (host [F] frames of current chunk n >= 0) exactly as
 * crc_bank_insert_poses does.  Scores are fp64 without FMA contraction, in the
 * order dx*dx+dy*dy+dz*dz, sqrt, /E; dot product left to right.
 *
 * Outputs (device):
 *   d_idx   [k] int32: the admissible chunks with the k smallest (s(j), j),
 *           ascending; slots r >= count hold the window-extension chunk of
 *           `p->ext_first` (or -1 when empty).
 *   d_score [k] fp64: s(j) for r < count, +inf otherwise.  May be NULL.
 *   d_count [1] int32: number of admissible chunks retrieved (<= k).
 * Then, for every CRC_SEG_RETRIEVED segment of `cache` with slot r < k and
 * d_idx[r] >= 0, keys [offset, offset+N_c) of every layer receive the K and V
 * of slab d_idx[r] % num_slabs (the gather), the keys re-positioned by `rope`
 * when it is not NULL.  Everything stays on the device.
 *
 * Every bank entry is scored once.  Banks of more than 512 entries are split over
 * several blocks whose candidates meet in `d_workspace`: device memory of at least
 * crc_retrieve_workspace_size(bank_count, k) bytes, 16-byte aligned, owned by the
 * caller and written by the call (its previous contents do not matter).  When that
 * size is 0 the workspace may be NULL.  One workspace serves one call at a time:
 * calls that may overlap on the GPU need workspaces of their own.
 * Enqueued work: a 4-byte memset of the workspace (when it is used), the scoring
 * launch and, with a cache, the gather launch.
 * Errors: CRC_ERR_INVALID_ARG (also a missing, short or misaligned workspace, a
 * non-finite E or w_v), CRC_ERR_SHAPE, CRC_ERR_UNSUPPORTED, CRC_ERR_CUDA.
 */
crc_status crc_retrieve(const crc_bank* bank, int32_t bank_count, const crc_shape* shape, const crc_frame* cur,
                        int32_t n, const crc_retrieval* p, const crc_cache* cache, const crc_rope* rope,
                        int32_t* d_idx, double* d_score, int32_t* d_count, void* d_workspace,
                        size_t workspace_bytes, cudaStream_t s);

/* Workspace bytes crc_retrieve needs for a bank of `bank_count` entries and k
 * slots: 0 up to 512 entries, else 16 bytes per (block of 512 entries, slot) plus
 * 256, rounded up (under 300 KB for any bank).  0 for invalid arguments. */
size_t crc_retrieve_workspace_size(int32_t bank_count, int32_t k);

/*
 * crc_retrieve_noalloc — crc_retrieve for callers that cannot allocate device memory.
 * (The paper has no counterpart: this is a deployment variant of the same call.)
 *
 * Who needs it: an engine's render thread with a fixed per-frame budget (cudaMalloc
 * and cudaFree can synchronise the device and take milliseconds), a plugin whose host
 * application owns all GPU memory, or a stream that must not fail half-way with an
 * out-of-memory error.  Instead of a caller workspace, banks of more than 512 entries
 * use a fixed scratch array inside the library's device code, CRC_NOALLOC_SCRATCH_BYTES
 * (64 KiB) on every GPU that loads the library, held until the process exits.  Nothing
 * is allocated or freed by the call.
 *
 * Arguments, results and errors are those of crc_retrieve, plus CRC_ERR_TOO_LARGE when
 * crc_retrieve_workspace_size(bank_count, k) exceeds the scratch (at k = 8 that is a
 * bank of more than 261 120 entries; at k = 1 no bank is too large), and CRC_ERR_CUDA
 * when the scratch's device address cannot be found.
 * The first call on each device that needs the scratch looks up its device address
 * (cudaGetSymbolAddress, once per device, with that device current); make that first
 * call before capturing any stream on that device.  Every call shares the one array,
 * which keeps the previous call's contents (each call clears what must start at zero):
 * calls that may overlap on the GPU -- on different streams, or from different host
 * threads -- race on it, so they must be ordered, e.g. on one stream.
 */
#define CRC_NOALLOC_SCRATCH_BYTES 65536
crc_status crc_retrieve_noalloc(const crc_bank* bank, int32_t bank_count, const crc_shape* shape,
                                const crc_frame* cur, int32_t n, const crc_retrieval* p, const crc_cache* cache,
                                const crc_rope* rope, int32_t* d_idx, double* d_score, int32_t* d_count,
                                cudaStream_t s);

/*
 * crc_gather — the gather half of crc_retrieve for a second cache that mirrors
 * the main one (Sec. 4.2 "Cache packing": the retrieved chunk is reinstated in
 * the control-branch cache too; that branch takes no correspondence bias).
 *
 *   pool      device [num_slabs][2][L][N_c][H][d] K (0) / V (1) slabs, dense, dtype
 *             of the call; chunk j lives in slab j % num_slabs.  The shape's L and
 *             H are those of the mirrored cache (e.g. the control blocks only).
 *   d_idx     device [k] int32 chunk of each retrieved slot, as written by
 *             crc_retrieve (negative = empty slot, left untouched).
 *   cache     every CRC_SEG_RETRIEVED segment with slot r < k and length N_c
 *             receives slab d_idx[r] % num_slabs; other keys are not touched.
 *   rope      NULL, or the re-positioning of the keys as for crc_retrieve.
 * Errors: CRC_ERR_INVALID_ARG (null pointers, k out of 1..CRC_MAX_K, bad rope),
 * CRC_ERR_SHAPE (cache strides, two segments for one slot), CRC_ERR_UNSUPPORTED
 * (alignment, rope layout), CRC_ERR_CUDA.
 */
crc_status crc_gather(const crc_shape* shape, const void* pool, int32_t num_slabs, const int32_t* d_idx, int32_t k,
                      const crc_cache* cache, const crc_rope* rope, cudaStream_t s);

/*
 * crc_correspond — Sec. 4.3, Eq. 3-4.  For every query token p = (t, i, j) of
 * the current chunk and every source frame s = r*F + f of retrieved slot r < k:
 *   X_t = z_p K_t^-1 (j, i, 1)^T,  X_s = R_s^T (R_t X_t + c_t - c_s),
 *   u^  = pi(K_s X_s),  cell = (floor(u^x + 1/2), floor(u^y + 1/2)),
 *   valid = z_p finite and > 0, u^ finite, [X_s]_z > 0, cell on the grid,
 *           [X_s]_z <= (1 + eps) D_s(cell)  (eps = +inf disables Eq. 4),
 *           d_idx[r] >= 0, and r < *d_count when d_count is not NULL
 *           (a window-extension slot is not a retrieval and gets no bias).
 * Source frames and depths are read from the bank at chunk d_idx[r] on the device.
 * The per-(frame, source frame) transform is composed in fp32 from the fp64 records
 * (camera-centre difference in fp64); per-token arithmetic is fp32.
 *
 *   cur      host [F] frames of the current chunk;  d_depth [F][h][w] fp32.
 *   d_uv     device [N_q][S][2] fp32 u^ (NaN where undefined), S = k*F.
 *   d_cell   device [N_q][S] int32: y*w + x, or -1 when not valid.  May be NULL.
 *   d_valid  device [N_q][S] uint8: 1 valid, 0 not.
 * Errors: CRC_ERR_INVALID_ARG; CRC_ERR_UNSUPPORTED when d_uv is not 8-byte aligned
 * or when the bank's depth array (capacity * F * h * w values) exceeds 2^31 - 1
 * values; CRC_ERR_CUDA.
 */
crc_status crc_correspond(const crc_shape* shape, const crc_frame* cur, const float* d_depth, const crc_bank* bank,
                          const int32_t* d_idx, const int32_t* d_count, int32_t k, float eps, float* d_uv,
                          int32_t* d_cell, uint8_t* d_valid, cudaStream_t s);

/* crc_biased_attention flags */
#define CRC_ATTN_DEFAULT 0
#define CRC_ATTN_SIMT 1      /* force the SIMT kernel (fp32 arithmetic) for any dtype */
#define CRC_ATTN_GAUSSIAN 2  /* opt-in: additive Gaussian bias lambda exp(-||u_k - u^||^2 / (2 sigma^2))
                                on the biased columns instead of Eq. 2's quadratic penalty
                                (a bonus that peaks at the correspondence).  bf16 with d = 128 runs
                                on the tensor-core kernel, which adds the bonus to each biased tile's
                                scores in the softmax; otherwise the SIMT kernel.  Not combined with
                                CRC_ATTN_SKIP_FAR, which is then ignored. */
#define CRC_ATTN_FRAME_CAUSAL 16  /* test mode of the block-causal reading: inside the current chunk
                                     (its CRC_SEG_CURRENT segment) a query of latent frame t sees
                                     only the keys of frames <= t; every other key stays visible */
#define CRC_ATTN_BIAS_DIRECT 8  /* tensor-core kernel, Eq. 2 form: evaluate the bias per score in the
                                   softmax (exact to fp32 rounding) even where the tensor-core
                                   expansion is within its error limit (see crc_biased_attention) */
#define CRC_ATTN_SKIP_FAR 4  /* opt-in approximation (tensor-core kernel, Eq. 2 form): a KV tile of a
                                retrieved frame is skipped for a block of 256 queries when every one of
                                them has a valid correspondence in that frame and the distance from the
                                box of those correspondences to the tile's key cells is at least
                                sigma sqrt(128 ln 2 / lambda), i.e. the bias scales each skipped weight by
                                at most 2^-64.  Only retrieved tiles are skipped, and only when the cache
                                has other active keys. */

/*
 * crc_biased_attention — Sec. 4.3, Eq. 2, for every layer l < L, head and query p:
 *   A_pk = q_p . k_k / sqrt(d) + lambda B(p, k),  O_p = sum_k softmax_k(A_pk) v_k
 *   B(p, k) = -||u_k - u^_s(p)||^2 / (2 sigma^2) when key k lies in a
 *             CRC_SEG_RETRIEVED segment of slot r, s = r*F + (position in the
 *             segment) / (h*w), u_k its (x, y) in that frame, and d_valid[p][s];
 *             0 for every other key (sink, window) and for invalid pairs.
 * Softmax runs over the active keys: keys inside a segment, minus retrieved slots
 * whose chunk is empty (d_slot_chunk[r] < 0, when d_slot_chunk is not NULL), and, with
 * CRC_ATTN_FRAME_CAUSAL, minus the current chunk's keys of frames after the query's
 * (query p lies in frame p / (h w); a key at position i of the CRC_SEG_CURRENT
 * segment in frame i / (h w)).
 * The bias is evaluated inside the tile loop and never stored.
 *
 *   q         [L][n_q][H][d] queries (dtype of the call); n_q = N_c.
 *   o         [L][n_q][H][d] output, same dtype.
 *   d_lse     device [L][H][n_q] fp32 natural-log sum-exp of the row, or NULL.
 *   d_uv, d_valid   correspondences [n_q][S] from crc_correspond (S = k*F).
 *   d_slot_chunk    device [k] int32 (crc_retrieve's d_idx) or NULL.
 *   d_status  device int32 or NULL: set non-zero if a kernel gave up waiting on
 *             an internal pipeline barrier (the output is then not valid).
 * bf16 (d = 128) runs on the tcgen05 tensor-core kernel with fp32 softmax and
 * accumulation, in either bias form; fp32 or CRC_ATTN_SIMT run the SIMT kernel in fp32.
 * Eq. 2 on the tensor-core kernel: the bias is added to S by the tensor core itself, as
 * a K = 16 extension of q.k (a rank-4 expansion of ||u_k - u^||^2 about the frame centre).
 * Its strength is taken to 16 significant bits (lambda scaled by 1 + delta, |delta| <=
 * 2^-17), and its terms cancel near the correspondence, so its error grows with the
 * grid: at most crc_bias_expansion_bound(lambda, sigma, h, w) = 2^-24 C (w^2 + h^2) in
 * base-2 logit units, C = lambda log2(e) / (2 sigma^2).  Where that exceeds 2^-9 (the
 * bf16 rounding of the softmax weights; e.g. lambda / sigma^2 > 5.39 on a 45 x 80 grid,
 * > 12.6 on 30 x 52) the kernel adds the bias per score in the softmax instead, exact to
 * fp32 rounding, at a lower throughput; CRC_ATTN_BIAS_DIRECT selects that everywhere.
 * The tensor-core kernel takes at most 640 KV tiles of 128 keys per call (each
 * segment is cut into tiles from its start, a retrieved segment per frame: up to
 * 81 920 keys) and h*w <= 65535; beyond that the call returns CRC_ERR_UNSUPPORTED
 * before any launch, and CRC_ATTN_SIMT takes it.
 * Errors: CRC_ERR_INVALID_ARG (also unknown flag bits), CRC_ERR_SHAPE,
 * CRC_ERR_UNSUPPORTED (dtype, d, alignment -- d_uv must be 8-byte aligned --, device
 * without sm_103a), CRC_ERR_CUDA.
 */
crc_status crc_biased_attention(const crc_shape* shape, crc_tensor q, const crc_cache* cache, crc_tensor o,
                                float* d_lse, int32_t n_q, const float* d_uv, const uint8_t* d_valid, int32_t k,
                                const int32_t* d_slot_chunk, float lambda, float sigma, int32_t flags,
                                int32_t* d_status, cudaStream_t s);

/* ---- a whole chunk step from a device-resident descriptor --------------------
 *
 * A chunk step of a stream (Sec. 4.2 "Cache layout" and "Loop-closure retrieval": one
 * step per generated chunk) is crc_cache_update, crc_retrieve, crc_correspond and
 * crc_biased_attention with values that change from step to step: the chunk index,
 * the window slot that receives the chunk, the fallback chunk, the re-positioning
 * target, which window segments hold a chunk yet, and the chunk's camera frames.
 * crc_chunk_step reads those from a descriptor in device memory, so that one captured
 * sequence of its launches (a CUDA graph) serves every step of the stream: the caller
 * rewrites the descriptor (for instance with a host-to-device copy captured in the
 * same graph, from a pinned buffer it rewrites before each replay) and replays. */

/* The per-step values, in device memory (8-byte aligned). */
typedef struct {
  int32_t n;               /* current chunk; the bank holds chunks 0..n (n < bank capacity)     */
  int32_t window_offset;   /* first cache key of the slot that receives chunk n (-1: none)      */
  int32_t ext_first;       /* crc_retrieval.ext_first of this step                              */
  int32_t rope_pos_slot0;  /* crc_rope.pos_slot0 of this step (unused without re-positioning)   */
  int32_t seg_length[CRC_MAX_SEGMENTS]; /* each cache segment's length this step, 0 ..
                                           its length in the plan (a retrieved one: 0 or N_c) */
  crc_frame frames[CRC_MAX_FRAMES];     /* the current chunk's frames (first F used)           */
} crc_step;

/* What stays fixed over the steps: every pointer is captured by the launches. */
typedef struct {
  crc_shape shape;
  crc_bank bank;             /* with its K/V slab pool                                        */
  crc_cache cache;           /* segment offsets, kinds, slots; lengths are the largest ones    */
  crc_retrieval retrieval;   /* ext_first is taken from the descriptor                        */
  crc_rope rope;             /* pairs = 0: no re-positioning; pos_slot0 from the descriptor    */
  float eps;                 /* Eq. 4 tolerance (INFINITY: off)                                */
  float lambda, sigma;       /* Eq. 2                                                          */
  int32_t attn_flags;        /* CRC_ATTN_* as for crc_biased_attention                         */
  /* per-step inputs, device, rewritten by the caller before each step */
  const float* d_depth;      /* [F][h][w] depth of chunk n                                     */
  const void* d_k;           /* [L][N_c][H][d] K and V of chunk n (dense)                       */
  const void* d_v;
  crc_tensor q;              /* [L][N_c][H][d] queries                                         */
  /* outputs, device */
  crc_tensor o;
  float* d_lse;              /* [L][H][N_c] or NULL                                            */
  int32_t* d_idx;            /* [k]                                                            */
  double* d_score;           /* [k] or NULL                                                    */
  int32_t* d_count;          /* [1]                                                            */
  float* d_uv;               /* [N_c][k F][2], 8-byte aligned                                   */
  int32_t* d_cell;           /* [N_c][k F] or NULL                                             */
  uint8_t* d_valid;          /* [N_c][k F]                                                     */
  int32_t* d_status;         /* [1], required: CRC_STEP_BAD_DESCRIPTOR when a kernel finds the
                                descriptor out of range (the bank and the cache are then left
                                untouched, the retrieval reports no chunk and the step's
                                outputs are not valid), or a timeout code of the attention kernel */
  void* d_workspace;         /* crc_retrieve_workspace_size(bank.capacity, k) bytes            */
  size_t workspace_bytes;
} crc_step_plan;

#define CRC_STEP_BAD_DESCRIPTOR 100

/*
 * crc_chunk_step — one chunk step with the per-step values of *d_step: the same
 * results, bit for bit, as crc_cache_update(bank, shape, n, frames, d_depth, d_k,
 * d_v, cache, window_offset), crc_retrieve over chunks 0..n (ext_first and the
 * re-positioning from the descriptor), crc_correspond and crc_biased_attention with
 * the descriptor's segment lengths, in that order on stream s.  Everything in the
 * plan is validated on the host; the descriptor is checked on the device (n within
 * the bank, the window slot within the cache, segment lengths within the plan's).
 * Enqueued work: the K/V and pose update, a 4-byte memset (when the retrieval
 * workspace is used), the scoring, the gather, the reprojection and the attention.
 * Errors: as the four calls, and CRC_ERR_INVALID_ARG for a missing status word,
 * descriptor or workspace.
 */
crc_status crc_chunk_step(const crc_step_plan* plan, const crc_step* d_step, cudaStream_t s);

/*
 * crc_host_copy — copies `bytes` bytes from src to dst with the GPU's SMs: how a
 * step's host-resident inputs (Q, the new chunk's K/V, its depth) reach the GPU and
 * its output O returns.  (The paper has no counterpart; Sec. 4.2-4.3 define the step
 * these copies feed.)
 *
 * On GB300 the GPU reaches page-locked host memory directly over the coherent CPU-GPU
 * link, so a kernel moves host data at the link's own rate (about 210 GB/s to the
 * device and 190 GB/s back, measured) without the copy engines; eight SMs suffice for
 * that rate.  On some machines the copy engines stall for 35-100 ms at a time;
 * copies issued by the SMs were not seen to stall.  The copy runs `blocks` blocks of
 * 1024 threads (0 = 8), each resident on one SM until it ends.  To run it beside a
 * kernel that fills the GPU, enqueue it on a stream of higher priority: at equal
 * priority its blocks wait until the earlier kernel has dispatched all of its own.
 *
 * src, dst: device memory of the current device, page-locked host memory (allocated
 *   or registered with CUDA) or managed memory, in any combination; both 16-byte
 *   aligned; the two ranges must not overlap.  bytes: any size.
 * Returns CRC_OK (0 bytes: nothing enqueued); CRC_ERR_INVALID_ARG for a null pointer,
 * blocks outside 0..4096, overlapping ranges, or a range the device cannot reach in
 * one contiguous mapping (pageable host memory, another device's memory, a range that
 * runs past its allocation into unmapped memory), all found before anything is
 * enqueued; CRC_ERR_UNSUPPORTED for a pointer that is not 16-byte aligned;
 * CRC_ERR_CUDA when the launch fails.
 */
crc_status crc_host_copy(void* dst, const void* src, size_t bytes, int32_t blocks, cudaStream_t s);

/* Bound on the error of the tensor-core expansion of the Eq. 2 bias on an h x w grid,
 * in base-2 logit units: 2^-24 lambda log2(e) / (2 sigma^2) (w^2 + h^2), besides the
 * consistent 2^-17 scale of the bias strength; +inf where
 * the key coordinates are not exact in bf16 (w or h above 256, or
 * (w-1)^2 + (h-1)^2 >= 2^16), which always takes the per-score form.  Host only. */
double crc_bias_expansion_bound(float lambda, float sigma, int32_t h, int32_t w);

#ifdef __cplusplus
}
#endif

#endif /* CRC_H_ */
