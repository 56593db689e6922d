// Biased flash attention on the 5th-generation tensor cores (Sec. 4.3, Eq. 2).
//
//   A_pk = q_p . k_k / sqrt(d) + lambda B_s(p, k),  B = -||u_k - u^_s(p)||^2 / (2 sigma^2)
//
// on retrieved-slot key columns with a valid correspondence, 0 elsewhere.  The
// bias is never written to memory: the tensor core adds it to S.  KV tiles are cut
// at every segment start and, inside retrieved segments, at every frame start, so
// that each tile has at most one source frame; a tile's ragged tail is masked the
// same way.  bf16 Q/K/V, fp32 scores, softmax and accumulation, bf16 O.
//
// Bias on the tensor core.  With coordinates relative to the frame centre
// (x' = x - (w-1)/2, y' = y - (h-1)/2) and A = lambda log2(e) / (2 sigma^2) in base-2
// units (0 when the pair is invalid), the bias of Eq. 2 expands as
//   A (q_k - 2 ux' x'_k - 2 uy' y'_k + ux'^2 + uy'^2),   q_k = x'_k^2 + y'_k^2,
// a dot product of a 4-vector per query row with a 4-vector per key.  A is rounded to
// two bf16 terms (A'), the other query coefficients are formed from A' in double-fp32
// arithmetic and split into four (linear terms) or three (constant term) bf16 terms,
// and q_k into two (exact: x', y' are half-integers), giving a K = 16 extension of the
// QK^T contraction whose products are exact:
//   query row: [ah ah al al | c1 c1 c1 c1 | c2 c2 c2 c2 | c3 c3 c3 | 1]
//   key row:   [qh ql qh ql | x' x' x' x' | y' y' y' y' | 1  1  1  | M]
// The last column masks keys past the tile's end (M = -2^100, else 0); an unbiased
// tile has zeros in the first fifteen key columns.  One extra tcgen05.mma
// (M = N = 128, K = 16, no-swizzle K-major operands) per query tile adds it to S,
// and the softmax never touches individual columns.
//
// Structure (one CTA = two 128-row query tiles of one (layer, head)):
//   warps 0-3   softmax of query tile 0   (TMEM lanes 0-127 of S0/O0)
//   warps 4-7   softmax of query tile 1   (TMEM lanes 0-127 of S1/O1)
//   warp  8     TMA producer: Q once, then K/V tiles of 128 keys, 2 stages each,
//               128-byte swizzled boxes of 128 rows x 64 elements
//   warp  9     TMEM owner and tcgen05.mma issuer (the warp converged, one elected lane)
//   warps 10-11 build, ahead of use, the key-side bias/mask operand of every tile
//               that needs one (3-deep ring; the producer declares a stage full only
//               once the tile's operand is built, and an MMA commit frees the slot)
// One FULL barrier per stage stands for K, V and the bias operand together, and one
// EMPTY barrier (a commit after the tile's last PV) frees the whole stage: the
// MMA warp waits once per KV tile for data, since issuing a 128 x 128 x 16 MMA
// occupies it for most of the time the tensor core runs it, and every wait or
// shared-memory load it makes costs it a round trip of issue time (which tiles
// carry a bias/mask operand it reads from a bit mask, 32 tiles a word).  The warp
// issues converged, one elected lane per instruction: measured, 39 clocks per MMA
// against 54 for a lone lane (50 against 110 while the other warps of its
// sub-partition run arithmetic).
// The query-side bias operand of each query tile is written by its own softmax
// warpgroup whenever the source frame of the next biased tile changes.
// TMEM (512 columns): S0 | S1 | O0 | O1, 128 fp32 columns each.  S = Q K^T is an
// SS MMA (both operands K-major in shared memory); each softmax thread reads its
// row of S, writes P in bf16 over the first 64 columns of the same S buffer and
// the MMA warp accumulates O += P V with P taken straight from TMEM (TS MMA, V
// MN-major in shared memory).  The MMA warp alternates the two query tiles, so
// the tensor core works on one tile while the other tile's softmax runs.
// Online softmax in base 2 with the row max kept stale until it grows by more
// than 2^8 (exact: the same max normalises P, O and the row sum); O in TMEM is
// rescaled only on those rare steps.  Keys outside every segment and retrieved
// slots without a chunk produce no tile at all.
//
// Accuracy of the expansion.  Its large terms (A q_k, 2 A ux' x'_k, ...) cancel to
// A d^2 near the correspondence, so its absolute error grows with the grid: in base-2
// logit units it stays below 2^-24 C (w^2 + h^2), C = lambda log2(e) / (2 sigma^2), on
// top of the consistent 2^-17 scale of A'.  With the coefficients formed in double-fp32
// their representation contributes 0.6-2.4 x 2^-28 C (w^2 + h^2) (a CPU model of these
// steps); this GPU measures 3.8-6.6 x 2^-28 C (w^2 + h^2) in all, the rest being the
// tensor core's own fp32 sum of the 16 products.  (Coefficients rounded to fp32 before
// the split measured 8-10 x 2^-28.)  The key terms are exact for grids up to 256 a
// side with (w-1)^2 + (h-1)^2 < 2^16.  Where the bound exceeds 2^-9 -- the bf16
// rounding of P -- or the grid is larger, the host selects the direct form (MODE =
// DIRECT): the K = 16 operand carries only the mask and the softmax adds C d^2 to
// every biased score from the key's cell, exact to fp32 rounding, at a lower throughput.
//
// The opt-in additive-Gaussian form (lambda exp(-d^2 / (2 sigma^2)) on the same
// columns) has no low-rank expansion either: its instantiation (MODE = GAUSS) adds
// the bonus to S in the softmax, column by column, before the row max.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>
#include <limits.h>
#include <math.h>
#include <string.h>

#include "internal.cuh"
#include "tc_ptx.cuh"

namespace crc {

namespace {

using namespace ptx;

constexpr int BM = 128;  // query rows per tile = TMEM lanes
constexpr int BN = 128;  // keys per KV tile
constexpr int HD = 128;  // head dim
constexpr int NQT = 2;   // query tiles per CTA
constexpr int ST = 2;    // stages for K and for V
constexpr int kThreads = 384;  // 3 warpgroups: softmax 0, softmax 1, producer/MMA/tables
constexpr int kWarpTma = 8;
constexpr int kWarpMma = 9;
// register split (setmaxnreg): the block launches with 384 x 168 registers; the
// producer warpgroup drops to 104 and each softmax warpgroup rises to 200:
// 2 x 128 x 200 + 128 x 104 = 384 x 168.
constexpr int kRegsSoftmax = 200;
constexpr int kRegsProducer = 104;
static_assert(2 * 128 * kRegsSoftmax + 128 * kRegsProducer <= kThreads * 168, "register split exceeds the launch");
constexpr int BOX = BM * 64 * 2;  // 128 rows x 64 bf16 = 16 KB
constexpr int TILE = 2 * BOX;     // 128 rows x 128 bf16 = 32 KB
constexpr int AUG = 128 * 16 * 2; // 128 rows x 16 bf16 bias operand = 4 KB
constexpr int kMaxTiles = 640;    // KV tiles per call (keys <= 81920)
constexpr int NBB = 3;            // ring of key-side bias/mask operands
// mbarrier wait policy per role (0 = poll; otherwise the suspend hint in ns)
constexpr uint32_t kHintSoftmax = 0;
constexpr uint32_t kHintMma = 0;
constexpr uint32_t kHintLoad = 0;
constexpr uint32_t kHintTable = 0;

constexpr int OFF_Q = 0;
constexpr int OFF_K = OFF_Q + NQT * TILE;
constexpr int OFF_V = OFF_K + ST * TILE;
constexpr int OFF_AQ = OFF_V + ST * TILE;      // query-side bias operand, one per query tile
constexpr int OFF_RB = OFF_AQ + NQT * AUG;     // key-side bias/mask operand ring
constexpr int OFF_TILES = OFF_RB + NBB * AUG;
constexpr int OFF_AMASK = OFF_TILES + kMaxTiles * 12;  // bit j: tile j is CLS_AUG
constexpr int OFF_BAR = OFF_AMASK + kMaxTiles / 8;
constexpr int NBAR = 1 + 2 * ST + 3 * NQT + 1 + NQT + 2 * NBB;
constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
constexpr int OFF_BOX = OFF_MISC + 64;  // per source frame: correspondence box of the CTA's queries
constexpr int SMEM_BYTES = OFF_BOX + CRC_MAX_K * CRC_MAX_FRAMES * 5 * 4 + 1024;  // + slack for 1024-byte alignment
static_assert(SMEM_BYTES <= 232448, "shared memory budget");

constexpr uint32_t TM_S = 0;    // S/P of tile x at column 128 x
constexpr uint32_t TM_O = 256;  // O of tile x at column 256 + 128 x
constexpr uint32_t TM_COLS = 512;

constexpr uint8_t CLS_PLAIN = 0;  // 128 active keys, no bias: Q K^T only
constexpr uint8_t CLS_AUG = 1;    // biased and/or ragged: Q K^T + bias/mask operand

struct TileInfo {
  uint32_t key0;    // first key of the tile
  uint8_t nact_m1;  // active keys - 1 (keys key0 .. key0 + nact - 1)
  uint8_t cls;
  int8_t s;         // source frame of the (biased) keys, -1 for an unbiased tile
  uint8_t kf1;      // current-chunk tiles: 1 + the keys' frame (frame-causal mask), else 0
  uint16_t q;       // ordinal among CLS_AUG tiles (ring position)
  uint16_t loc0;    // index of key0 inside its source frame (biased tiles)
};

struct TcParams {
  AttnArgs a;
  float scale_log2;  // log2(e) / sqrt(d)
  float coef_log2;   // -lambda log2(e) / (2 sigma^2)
  float gauss_gc;    // additive-Gaussian form: lambda sqrt(d), the bonus at d = 0 in raw score units
  float gauss_k;     // and log2(e) / (2 sigma^2), so that the bonus is gauss_gc 2^(-d^2 gauss_k)
  uint64_t timeout_ns;
};

// barrier indices
// FULL(s): K, V and (for a biased or ragged tile) the key-side bias/mask operand of
// stage s are in shared memory.  EMPTY(s): the stage's last MMA (PV of tile 1) retired.
__device__ __forceinline__ int B_QFULL() { return 0; }
__device__ __forceinline__ int B_FULL(int s) { return 1 + s; }
__device__ __forceinline__ int B_EMPTY(int s) { return 1 + ST + s; }
__device__ __forceinline__ int B_SFULL(int x) { return 1 + 2 * ST + x; }
__device__ __forceinline__ int B_PREADY(int x) { return 1 + 2 * ST + NQT + x; }
__device__ __forceinline__ int B_OFINAL(int x) { return 1 + 2 * ST + 2 * NQT + x; }
__device__ __forceinline__ int B_DRAIN() { return 1 + 2 * ST + 3 * NQT; }
__device__ __forceinline__ int B_AREADY(int x) { return 2 + 2 * ST + 3 * NQT + x; }
__device__ __forceinline__ int B_BFULL(int b) { return 2 + 2 * ST + 4 * NQT + b; }
__device__ __forceinline__ int B_BEMPTY(int b) { return 2 + 2 * ST + 4 * NQT + NBB + b; }

// ---- packed fp32 pairs (Blackwell f32x2 ALU ops) and three-input max ----------
__device__ __forceinline__ uint64_t pk2(float a, float b) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
  return r;
}
__device__ __forceinline__ void upk2(uint64_t r, float& a, float& b) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(r));
}
__device__ __forceinline__ uint64_t ffma2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t fadd2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ float max3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__device__ __forceinline__ uint32_t bf16_bits(float v) {
  return (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn(v));
}
// Error-free transformations in fp32: each operation rounded once, nothing contracted.
__device__ __forceinline__ void two_prod(float a, float b, float& p, float& e) {  // a b = p + e exactly
  p = __fmul_rn(a, b);
  e = __fmaf_rn(a, b, -p);
}
__device__ __forceinline__ void two_sum(float a, float b, float& s, float& e) {  // a + b = s + e exactly
  s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}
// hi + lo (|lo| well below |hi|) as N bf16 terms, each the nearest bf16 to what remains;
// lo joins the remainder after the first term.  The remainder after term i is exact in
// fp32, so the error is the one rounding that folds lo in (2^-32 of hi) plus what the
// last term leaves (2^-26 of hi for N = 3, 2^-35 for N = 4).
template <int N>
__device__ __forceinline__ void split_df(float hi, float lo, uint32_t (&t)[N]) {
  float r = hi;
#pragma unroll
  for (int i = 0; i < N; ++i) {
    const __nv_bfloat16 b = __float2bfloat16_rn(r);
    t[i] = (uint32_t)__bfloat16_as_ushort(b);
    r = __fsub_rn(r, __bfloat162float(b));
    if (i == 0) r = __fadd_rn(r, lo);
  }
}
// Write one 16-element bf16 row (given as 8 packed words) of a no-swizzle K-major
// 128 x 16 operand: 8-row x 16-byte core matrices, K halves 128 bytes apart,
// 8-row groups 256 bytes apart.
__device__ __forceinline__ void store_aug_row(uint8_t* base, int row, const uint32_t (&w)[8]) {
  uint8_t* p = base + (row >> 3) * 256 + (row & 7) * 16;
  *reinterpret_cast<uint4*>(p) = make_uint4(w[0], w[1], w[2], w[3]);
  *reinterpret_cast<uint4*>(p + 128) = make_uint4(w[4], w[5], w[6], w[7]);
}

// One query row's correspondences in the two source frames of a KV tile, with the
// bias coefficient already zero for invalid pairs (exact fallback).
struct Corr {
  float uxA, uyA, cA;
};

__device__ __forceinline__ Corr load_corr(const AttnArgs& a, const TileInfo* tiles, int j, int nt, int p, bool row_ok,
                                          float coef) {
  Corr c{0.f, 0.f, 0.f};
  if (j >= nt || !row_ok) return c;
  const TileInfo ti = tiles[j];
  if (ti.s < 0) return c;
  const int64_t ia = (int64_t)p * a.S + ti.s;
  if (__ldg(a.valid + ia)) {
    const float2 u = __ldg(reinterpret_cast<const float2*>(a.uv) + ia);
    c.uxA = u.x;
    c.uyA = u.y;
    c.cA = coef;
  }
  return c;
}

// Query-side bias operand row for source frame A of `c` (raw score units).  The bias
// strength is taken as A' = two bf16 terms of A (16 bits; A' = A (1 + delta), |delta| <=
// 2^-17, a consistent scale of the whole bias) and every coefficient is formed from A' in
// double-fp32 arithmetic before its split: -2 A' ux' and -2 A' uy' into four bf16 terms,
// A' (ux'^2 + uy'^2) into three.
//   query row: [ah ah al al | c1 c1 c1 c1 | c2 c2 c2 c2 | c3 c3 c3 | 1]
//   key row:   [qh ql qh ql | x' x' x' x' | y' y' y' y' | 1  1  1  | M]
__device__ __forceinline__ void aug_query_row(const Corr& c, float xc, float yc, float inv_sc, uint32_t (&w)[8]) {
  const float A = __fmul_rn(c.cA, inv_sc);
  const __nv_bfloat16 ah = __float2bfloat16_rn(A);
  const float ahf = __bfloat162float(ah);
  const __nv_bfloat16 al = __float2bfloat16_rn(__fsub_rn(A, ahf));
  const float alf = __bfloat162float(al);
  const float ux = __fsub_rn(c.uxA, xc), uy = __fsub_rn(c.uyA, yc);
  float p, e;
  uint32_t t1[4], t2[4], t3[3];
  // -2 A' u = -2 (ah u + al u): the first product exactly, the second (2^-9 of it) rounded once
  two_prod(ahf, ux, p, e);
  split_df<4>(-2.f * p, -2.f * __fmaf_rn(alf, ux, e), t1);
  two_prod(ahf, uy, p, e);
  split_df<4>(-2.f * p, -2.f * __fmaf_rn(alf, uy, e), t2);
  // A' (ux^2 + uy^2), the sum of squares carried as two fp32 terms
  float sx, ex, sy, ey, sq, es;
  two_prod(ux, ux, sx, ex);
  two_prod(uy, uy, sy, ey);
  two_sum(sx, sy, sq, es);
  const float sl = __fadd_rn(__fadd_rn(ex, ey), es);
  two_prod(ahf, sq, p, e);
  split_df<3>(p, __fmaf_rn(ahf, sl, __fmaf_rn(alf, sq, e)), t3);
  const uint32_t hb = (uint32_t)__bfloat16_as_ushort(ah), lb = (uint32_t)__bfloat16_as_ushort(al);
  w[0] = hb | (hb << 16);
  w[1] = lb | (lb << 16);
  w[2] = t1[0] | (t1[1] << 16);
  w[3] = t1[2] | (t1[3] << 16);
  w[4] = t2[0] | (t2[1] << 16);
  w[5] = t2[2] | (t2[3] << 16);
  w[6] = t3[0] | (t3[1] << 16);
  w[7] = t3[2] | (bf16_bits(1.f) << 16);  // mask column
}

// fp32 <-> int keys with the same order, for shared-memory atomic min / max
__device__ __forceinline__ int ord_key(float f) {
  const int b = __float_as_int(f);
  return b >= 0 ? b : b ^ 0x7fffffff;
}
__device__ __forceinline__ float ord_val(int k) { return __int_as_float(k >= 0 ? k : k ^ 0x7fffffff); }

__device__ __forceinline__ void fail(const TcParams& P, volatile int* abort_flag, int code) {
  *abort_flag = 1;
  if (P.a.status) atomicExch(P.a.status, code);
}

}  // namespace

// How the bias reaches S: the Eq. 2 expansion on the tensor core, or per score in
// the softmax (Eq. 2 directly, or the opt-in additive-Gaussian form).
constexpr int kBiasTensor = 0;
constexpr int kBiasGauss = 1;
constexpr int kBiasDirect = 2;

// MODE: one of the kBias* forms; the tensor-core instantiation carries none of the
// per-score code.  FC: the frame-causal test mode (CRC_ATTN_FRAME_CAUSAL), compiled
// only into its own instantiations (its per-tile test cost the default kernel 1 %).
template <int MODE, bool FC>
__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                   const __grid_constant__ CUtensorMap tmV, const __grid_constant__ TcParams P) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  const AttnArgs& a = P.a;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int q0 = blockIdx.x * NQT * BM;
  const int head = blockIdx.y, layer = blockIdx.z;
  auto bar = [&](int i) { return sbase + OFF_BAR + 8u * (uint32_t)i; };
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + OFF_MISC);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + OFF_MISC + 4);
  int* ntiles_slot = reinterpret_cast<int*>(smem + OFF_MISC + 8);
  TileInfo* tiles = reinterpret_cast<TileInfo*>(smem + OFF_TILES);
  const float xc = 0.5f * (float)(a.w - 1), yc = 0.5f * (float)(a.h - 1);

  if (tid == 0) {
    mbar_init(bar(B_QFULL()), 1);
    for (int s = 0; s < ST; ++s) {
      mbar_init(bar(B_FULL(s)), 1);
      mbar_init(bar(B_EMPTY(s)), 1);
    }
    for (int x = 0; x < NQT; ++x) {
      mbar_init(bar(B_SFULL(x)), 1);
      mbar_init(bar(B_PREADY(x)), BM);
      mbar_init(bar(B_OFINAL(x)), 1);
      mbar_init(bar(B_AREADY(x)), BM);
    }
    mbar_init(bar(B_DRAIN()), 1);
    for (int b = 0; b < NBB; ++b) {
      mbar_init(bar(B_BFULL(b)), 2);   // the two table warps
      mbar_init(bar(B_BEMPTY(b)), 1);  // a tcgen05.commit after the tile's last MMA
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  // CRC_ATTN_SKIP_FAR: per source frame, whether every query of this CTA has a valid
  // correspondence there, and the bounding box of those correspondences
  int* box = reinterpret_cast<int*>(smem + OFF_BOX);  // [S][5]: x min, x max, y min, y max, all valid
  const bool skip_far = a.skip_far != 0;
  if (skip_far) {
    for (int i = tid; i < a.S; i += kThreads) {
      box[5 * i + 0] = INT_MAX;
      box[5 * i + 1] = INT_MIN;
      box[5 * i + 2] = INT_MAX;
      box[5 * i + 3] = INT_MIN;
      box[5 * i + 4] = 1;
    }
    __syncthreads();
    const int rows = min(NQT * BM, a.Nq - q0);
    for (int e = tid; e < rows * a.S; e += kThreads) {
      const int rr = e / a.S, sf = e - rr * a.S;
      const int64_t pi = (int64_t)(q0 + rr) * a.S + sf;
      if (!a.valid[pi]) {
        atomicAnd(&box[5 * sf + 4], 0);
        continue;
      }
      const float2 u = reinterpret_cast<const float2*>(a.uv)[pi];
      atomicMin(&box[5 * sf + 0], ord_key(u.x));
      atomicMax(&box[5 * sf + 1], ord_key(u.x));
      atomicMin(&box[5 * sf + 2], ord_key(u.y));
      atomicMax(&box[5 * sf + 3], ord_key(u.y));
    }
    __syncthreads();
  }
  if (warp == 0) {
    // KV tiles: each segment is cut into tiles of 128 keys from its start; retrieved
    // segments are cut per source frame, so that a tile has at most one frame
    const int hw = a.h * a.w;
    uint32_t* amask = reinterpret_cast<uint32_t*>(smem + OFF_AMASK);
    for (int i = lane; i < kMaxTiles / 32; i += 32) amask[i] = 0u;
    __syncwarp();
    int count = 0, qa = 0;
    for (int g = 0; g < a.nseg; ++g) {
      const crc_segment sg = a.seg[g];
      const int len = seg_length(a, g);
      if (len <= 0) continue;
      const bool ret = sg.kind == CRC_SEG_RETRIEVED;
      // the current chunk's segment is cut per frame too when the frame-causal mask is on
      const bool curc = FC && sg.kind == CRC_SEG_CURRENT;
      if (ret && a.slot_chunk && a.slot_chunk[sg.slot] < 0) continue;  // empty slot: masked
      const int nr = (ret || curc) ? a.F : 1;
      for (int rr = 0; rr < nr; ++rr) {
        const int rstart = (ret || curc) ? sg.offset + rr * hw : sg.offset;
        const int rlen = (ret || curc) ? hw : len;
        const int ntile = (rlen + BN - 1) / BN;
        for (int base = 0; base < ntile; base += 32) {
          const int t = base + lane;
          const bool act = t < ntile;
          TileInfo ti;
          const int nact = act ? min(BN, rlen - t * BN) : 1;
          ti.key0 = (uint32_t)(rstart + t * BN);
          ti.nact_m1 = (uint8_t)(nact - 1);
          ti.s = ret ? (int8_t)(sg.slot * a.F + rr) : (int8_t)-1;
          ti.cls = (nact == BN && !ret) ? CLS_PLAIN : CLS_AUG;
          ti.kf1 = curc ? (uint8_t)(rr + 1) : 0;
          ti.loc0 = (uint16_t)(t * BN);
          bool keep = act;
          if (skip_far && ret && act) {
            // the tile's key cells against the box of this frame's correspondences
            const int sf = sg.slot * a.F + rr;
            if (box[5 * sf + 4] && box[5 * sf + 0] != INT_MAX) {
              const int l0 = t * BN, l1 = l0 + nact - 1;
              const int y0 = l0 / a.w, y1 = l1 / a.w;
              const float kx0 = y0 == y1 ? (float)(l0 - y0 * a.w) : 0.f;
              const float kx1 = y0 == y1 ? (float)(l1 - y1 * a.w) : (float)(a.w - 1);
              const float dx = fmaxf(0.f, fmaxf(ord_val(box[5 * sf + 0]) - kx1, kx0 - ord_val(box[5 * sf + 1])));
              const float dy = fmaxf(0.f, fmaxf(ord_val(box[5 * sf + 2]) - (float)y1, (float)y0 - ord_val(box[5 * sf + 3])));
              keep = !(dx * dx + dy * dy >= a.skip_d2);
            }
          }
          const unsigned lt = (1u << lane) - 1u;
          const unsigned m = __ballot_sync(0xffffffffu, keep);
          const unsigned ma = __ballot_sync(0xffffffffu, keep && ti.cls == CLS_AUG);
          ti.q = (uint16_t)(qa + __popc(ma & lt));
          if (keep) {
            const int ti_idx = count + __popc(m & lt);
            tiles[ti_idx] = ti;
            if (ti.cls == CLS_AUG) atomicOr(&amask[ti_idx >> 5], 1u << (ti_idx & 31));
          }
          count += __popc(m);
          qa += __popc(ma);
        }
      }
    }
    if (lane == 0) *ntiles_slot = count;
  }
  if (warp == kWarpMma) {
    tmem_alloc(smem_u32(tmem_slot), TM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const int nt = *ntiles_slot;
  const uint64_t T = P.timeout_ns;

  if (warp >= 8) {
   asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;\n" ::"n"(kRegsProducer));
   if (warp == kWarpTma) {
    // ------------------------------------------------------------ producer
    if (lane == 0 && nt > 0) {
      prefetch_tensormap(&tmQ);
      prefetch_tensormap(&tmK);
      prefetch_tensormap(&tmV);
      mbar_arrive_expect_tx(bar(B_QFULL()), NQT * TILE);
      for (int x = 0; x < NQT; ++x)
        for (int b = 0; b < 2; ++b)
          tma_load_4d(sbase + OFF_Q + x * TILE + b * BOX, &tmQ, bar(B_QFULL()), b * 64, head, q0 + x * BM, layer);
      // one full barrier per stage covers K, V and the tile's bias/mask operand, so
      // that the MMA issuer waits once per KV tile
      int issued = 0;
      for (int j = 0; j < nt; ++j) {
        const int st = j % ST;
        const uint32_t par = ((j / ST) & 1) ^ 1;
        const TileInfo ti = tiles[j];
        if (!mbar_wait(bar(B_EMPTY(st)), par, abort_flag, T, kHintLoad)) {
          fail(P, abort_flag, 1);
          break;
        }
        if (ti.cls == CLS_AUG &&
            !mbar_wait(bar(B_BFULL(ti.q % NBB)), (ti.q / NBB) & 1, abort_flag, T, kHintLoad)) {
          fail(P, abort_flag, 2);
          break;
        }
        mbar_arrive_expect_tx(bar(B_FULL(st)), 2 * TILE);
        for (int b = 0; b < 2; ++b)
          tma_load_4d(sbase + OFF_K + st * TILE + b * BOX, &tmK, bar(B_FULL(st)), b * 64, head, (int)ti.key0, layer);
        for (int b = 0; b < 2; ++b)
          tma_load_4d(sbase + OFF_V + st * TILE + b * BOX, &tmV, bar(B_FULL(st)), b * 64, head, (int)ti.key0, layer);
        issued = j + 1;
      }
      if (*abort_flag) {
        // let the copies already issued land before the CTA can exit
        const uint64_t lim = 100000000ull;
        volatile int never = 0;
        mbar_wait(bar(B_QFULL()), 0, &never, lim);
        for (int j = (issued > ST ? issued - ST : 0); j < issued; ++j)
          mbar_wait(bar(B_FULL(j % ST)), (j / ST) & 1, &never, lim);
      }
    }
   } else if (warp > kWarpMma) {
    // ------------------------------------------------------------ tables
    // Warps 10-11 (64 threads, two keys each) build the key-side bias/mask operand
    // of every CLS_AUG tile ahead of the MMA warp.
    const int bt = tid - (kWarpMma + 1) * 32;
    const uint32_t one = bf16_bits(1.f), neg = bf16_bits(-0x1p100f);
    for (int j = 0; j < nt; ++j) {
      const TileInfo ti = tiles[j];
      if (ti.cls != CLS_AUG) continue;
      const int b = ti.q % NBB;
      if (!mbar_wait(bar(B_BEMPTY(b)), ((ti.q / NBB) & 1) ^ 1, abort_flag, T, kHintTable)) {
        fail(P, abort_flag, 9);
        break;
      }
      uint8_t* blk = smem + OFF_RB + b * AUG;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int row = 2 * bt + h;
        const uint32_t mask = row <= (int)ti.nact_m1 ? 0u : neg;
        uint32_t w[8] = {0u, 0u, 0u, 0u, 0u, 0u, 0u, mask << 16};
        if (ti.s >= 0 && MODE == kBiasTensor) {
          // grid cell of the key inside its source frame, relative to the frame centre
          const int loc = (int)ti.loc0 + row;
          const int yi = loc / a.w;
          const float xr = (float)(loc - yi * a.w) - xc, yr = (float)yi - yc;
          const float q = fmaf(xr, xr, yr * yr);
          const uint32_t qh = bf16_bits(q);
          const uint32_t ql = bf16_bits(q - __bfloat162float(__ushort_as_bfloat16((unsigned short)qh)));
          const uint32_t xb = bf16_bits(xr), yb = bf16_bits(yr);
          w[0] = qh | (ql << 16);  // [qh ql qh ql | x' x4 | y' x4 | 1 1 1 | M]
          w[1] = w[0];
          w[2] = xb | (xb << 16);
          w[3] = w[2];
          w[4] = yb | (yb << 16);
          w[5] = w[4];
          w[6] = one | (one << 16);
          w[7] = one | (mask << 16);
        }
        store_aug_row(blk, row, w);
      }
      fence_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(B_BFULL(b)));
    }
   } else if (warp == kWarpMma) {
    // ------------------------------------------------------------ MMA issuer
    // The whole warp runs this loop, converged, and one elected lane issues each
    // MMA and commit; every wait's outcome is made warp-uniform before it is used.
    if (nt > 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(BM, BN, 0, 0);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(BM, HD, 0, 1);
      // descriptors of the operand bases; advancing along K adds (bytes >> 4) to the
      // start-address field, which cannot carry out of its 14 bits for shared memory
      const uint64_t dq0 = sdesc_sw128(sbase + OFF_Q, 16, 1024);
      const uint64_t dk0 = sdesc_sw128(sbase + OFF_K, 16, 1024);
      const uint64_t dv0 = sdesc_sw128(sbase + OFF_V, BOX, 1024);
      const uint64_t daq0 = sdesc_none(sbase + OFF_AQ, 128, 256);
      const uint64_t dbk0 = sdesc_none(sbase + OFF_RB, 128, 256);
      auto issue_qk = [&](int x, int st, bool aug, int bs) {
        const uint64_t ad = dq0 + (uint64_t)((x * TILE) >> 4);
        const uint64_t bd = dk0 + (uint64_t)((st * TILE) >> 4);
        const uint32_t d = tmem + TM_S + 128u * x;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const uint64_t off = (uint64_t)(((kk >> 2) * BOX + (kk & 3) * 32) >> 4);
          mma_ss_elect(d, ad + off, bd + off, idesc_qk, kk > 0 ? 1u : 0u);
        }
        if (aug)  // + bias/mask: query-side x key-side operand, K = 16
          mma_ss_elect(d, daq0 + (uint64_t)((x * AUG) >> 4), dbk0 + (uint64_t)((bs * AUG) >> 4), idesc_qk, 1u);
      };
      auto issue_pv = [&](int x, int st, bool acc) {
        const uint64_t bd = dv0 + (uint64_t)((st * TILE) >> 4);
        const uint32_t d = tmem + TM_O + 128u * x;
        const uint32_t pa = tmem + TM_S + 128u * x;
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk)
          mma_ts_elect(d, pa + 8u * kk, bd + (uint64_t)((kk * 2048) >> 4), idesc_pv, (acc || kk > 0) ? 1u : 0u);
      };
      // query tile 1 may hold no query at all (the last CTA of a head); then only
      // tile 0's MMAs run, and they release the stages and bias operands
      const bool live1 = q0 + BM < a.Nq;
      // Which tiles carry the bias/mask operand comes from a bit mask, one shared-memory
      // word per 32 tiles, and their ring slots from a running count: every load the
      // warp waits on holds up its MMA issue for a shared-memory round trip.
      const uint32_t* amask = reinterpret_cast<const uint32_t*>(smem + OFF_AMASK);
      uint32_t amw = amask[0];
      const bool aug0 = (amw & 1u) != 0;
      int bnext = aug0 ? 1 % NBB : 0;
      bool ok = mbar_wait(bar(B_QFULL()), 0, abort_flag, T) && mbar_wait(bar(B_FULL(0)), 0, abort_flag, T) &&
                mbar_wait(bar(B_AREADY(0)), 0, abort_flag, T) &&
                (!live1 || mbar_wait(bar(B_AREADY(1)), 0, abort_flag, T));
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) fail(P, abort_flag, 3);
      if (ok) {
        tc_fence_after();
        issue_qk(0, 0, aug0, 0);
        mma_commit_elect(bar(B_SFULL(0)));
        if (live1) {
          issue_qk(1, 0, aug0, 0);
          mma_commit_elect(bar(B_SFULL(1)));
        }
        if (aug0) mma_commit_elect(bar(B_BEMPTY(0)));
        // tile 0 alone: its MMAs release every stage and bias operand
        for (int j = 0; j < nt && ok && !live1; ++j) {
          const int st = j % ST;
          const int jn = j + 1, stn = jn % ST;
          const bool more = jn < nt;
          if (more && (jn & 31) == 0) amw = amask[jn >> 5];
          const bool augn = more && ((amw >> (jn & 31)) & 1u) != 0;
          const int bs = bnext;
          if (augn) bnext = bnext + 1 == NBB ? 0 : bnext + 1;
          ok = __all_sync(0xffffffffu, mbar_wait(bar(B_PREADY(0)), j & 1, abort_flag, T, kHintMma));
          if (!ok) { fail(P, abort_flag, 4); break; }
          tc_fence_after();
          issue_pv(0, st, j > 0);
          mma_commit_elect(bar(B_EMPTY(st)));
          if (more) {
            ok = __all_sync(0xffffffffu, mbar_wait(bar(B_FULL(stn)), (jn / ST) & 1, abort_flag, T, kHintMma));
            if (!ok) { fail(P, abort_flag, 5); break; }
            tc_fence_after();
            issue_qk(0, stn, augn, bs);
            mma_commit_elect(bar(B_SFULL(0)));
            if (augn) mma_commit_elect(bar(B_BEMPTY(bs)));
          } else {
            mma_commit_elect(bar(B_OFINAL(0)));
          }
        }
        // both tiles, interleaved on the tensor core
        for (int j = 0; j < nt && ok && live1; ++j) {
          const int st = j % ST;
          const int jn = j + 1, stn = jn % ST;
          const bool more = jn < nt;
          if (more && (jn & 31) == 0) amw = amask[jn >> 5];
          const bool augn = more && ((amw >> (jn & 31)) & 1u) != 0;
          const int bs = bnext;
          if (augn) bnext = bnext + 1 == NBB ? 0 : bnext + 1;
          ok = __all_sync(0xffffffffu, mbar_wait(bar(B_PREADY(0)), j & 1, abort_flag, T, kHintMma));
          if (!ok) { fail(P, abort_flag, 4); break; }
          tc_fence_after();
          issue_pv(0, st, j > 0);
          if (more) {
            ok = __all_sync(0xffffffffu, mbar_wait(bar(B_FULL(stn)), (jn / ST) & 1, abort_flag, T, kHintMma));
            if (!ok) { fail(P, abort_flag, 5); break; }
            tc_fence_after();
            issue_qk(0, stn, augn, bs);
            mma_commit_elect(bar(B_SFULL(0)));
          } else {
            mma_commit_elect(bar(B_OFINAL(0)));
          }
          ok = __all_sync(0xffffffffu, mbar_wait(bar(B_PREADY(1)), j & 1, abort_flag, T, kHintMma));
          if (!ok) { fail(P, abort_flag, 6); break; }
          tc_fence_after();
          issue_pv(1, st, j > 0);
          mma_commit_elect(bar(B_EMPTY(st)));
          if (more) {
            issue_qk(1, stn, augn, bs);
            mma_commit_elect(bar(B_SFULL(1)));
            if (augn) mma_commit_elect(bar(B_BEMPTY(bs)));
          } else {
            mma_commit_elect(bar(B_OFINAL(1)));
          }
        }
      }
      // every MMA issued so far has retired once this barrier fires
      volatile int never = 0;
      mma_commit_elect(bar(B_DRAIN()));
      mbar_wait(bar(B_DRAIN()), 0, &never, 100000000ull);
    }
   }
  } else {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;\n" ::"n"(kRegsSoftmax));
    // ------------------------------------------------------------ softmax
    const int x = warp >> 2;          // query tile
    const int wq = warp & 3;          // TMEM lane quarter
    const int r = wq * 32 + lane;     // row in tile = TMEM lane
    const int p = q0 + x * BM + r;    // query index
    if (q0 + x * BM < a.Nq) {         // else: a query tile without any query, no MMA runs for it
    const bool row_ok = p < a.Nq;
    const int qframe = p / (a.h * a.w);  // the query's latent frame (frame-causal mode)
    const uint32_t trow = tmem + ((uint32_t)(wq * 32) << 16);
    const uint32_t tS = trow + TM_S + 128u * x;
    const uint32_t tO = trow + TM_O + 128u * x;
    uint8_t* aq = smem + OFF_AQ + x * AUG;
    // scores are in raw units z = q.k (+ bias / scale); one FMA per element maps
    // them to log2 units for the exponent: p = 2^(z * sc - m)
    const float sc = P.scale_log2;
    const float inv_sc = 1.f / sc;
    const uint64_t SC2 = pk2(sc, sc);
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    // per-row correspondence of the (at most two) source frames of a tile,
    // loaded one tile ahead so that the global-load latency overlaps a tile
    Corr nxt = load_corr(a, tiles, 0, nt, p, row_ok, P.coef_log2);
    // query-side bias/mask operand: the first tile's source frame (or no bias).  In
    // the per-score forms it carries only the mask multiplier, and the bias is added
    // to S in the softmax from the current frame's correspondence `cur`.
    constexpr bool gauss = MODE != kBiasTensor;
    const Corr none{0.f, 0.f, 0.f};
    int aug_frame = nt > 0 ? tiles[0].s : -1;
    Corr cur = nxt;
    {
      uint32_t w[8];
      aug_query_row(gauss ? none : nxt, xc, yc, inv_sc, w);
      store_aug_row(aq, r, w);
      fence_async_smem();
    }
    mbar_arrive(bar(B_AREADY(x)));
    for (int j = 0; j < nt; ++j) {
      // the next tile's source frame; its correspondence is fetched (a tile ahead, so
      // that the global-load latency overlaps this tile) only when the query-side
      // bias operand has to change for it
      int8_t s_next = -1;
      if (j + 1 < nt) {
        const TileInfo tn = tiles[j + 1];
        if (tn.cls == CLS_AUG && tn.s >= 0 && tn.s != aug_frame) s_next = tn.s;
      }
      if (s_next >= 0) nxt = load_corr(a, tiles, j + 1, nt, p, row_ok, P.coef_log2);
      if (ok && !mbar_wait(bar(B_SFULL(x)), j & 1, abort_flag, T, kHintSoftmax)) { fail(P, abort_flag, 7); ok = false; }
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      tc_fence_after();
      uint32_t sr[128];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(tS + 32u * c, *reinterpret_cast<uint32_t(*)[32]>(&sr[32 * c]));
      tmem_wait_ld();
      if constexpr (MODE != kBiasTensor) {
        // per-score bias for a biased tile and a valid correspondence, with d the grid
        // distance from the key's cell (x, y), walked column by column, to u^ of the
        // tile's source frame:
        //   GAUSS:  S += lambda sqrt(d) 2^(-d^2 log2(e) / (2 sigma^2))
        //   DIRECT: S += (C / scale) d^2, Eq. 2 in raw score units (C < 0)
        const TileInfo tj = tiles[j];
        if (tj.s >= 0 && cur.cA != 0.f) {
          const int y0 = (int)tj.loc0 / a.w;
          float xf = (float)((int)tj.loc0 - y0 * a.w), yf = (float)y0;
          const float wf = (float)a.w, gk = P.gauss_k, gc = P.gauss_gc;
          const float araw = cur.cA * inv_sc;
          float dy = cur.uyA - yf;
          float dy2 = MODE == kBiasGauss ? dy * dy * gk : dy * dy;
#pragma unroll
          for (int c = 0; c < 128; ++c) {
            const float dx = cur.uxA - xf;
            if constexpr (MODE == kBiasGauss) {
              const float g = ex2(-fmaf(dx * dx, gk, dy2));
              sr[c] = __float_as_uint(fmaf(gc, g, __uint_as_float(sr[c])));
            } else {
              sr[c] = __float_as_uint(fmaf(araw, fmaf(dx, dx, dy2), __uint_as_float(sr[c])));
            }
            xf += 1.f;
            if (xf == wf) {
              xf = 0.f;
              yf += 1.f;
              dy = cur.uyA - yf;
              dy2 = MODE == kBiasGauss ? dy * dy * gk : dy * dy;
            }
          }
        }
      }
      // frame-causal mode: a tile of the current chunk's frame f is invisible to this row when
      // the row's query frame is earlier; its weights are then 2^-inf = 0 and m, l stay put
      bool rowmask = false;
      if constexpr (FC) {
        const int kf1 = tiles[j].kf1;
        rowmask = kf1 > 0 && kf1 - 1 > qframe;
      }
      // row max: eight running three-input max chains, then a final fold
      float mx[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) mx[i] = fmaxf(__uint_as_float(sr[i]), __uint_as_float(sr[8 + i]));
#pragma unroll
      for (int c = 16; c < 128; c += 16)
#pragma unroll
        for (int i = 0; i < 8; ++i) mx[i] = max3f(mx[i], __uint_as_float(sr[c + i]), __uint_as_float(sr[c + 8 + i]));
      const float mt = rowmask ? -INFINITY
                               : max3f(max3f(mx[0], mx[1], mx[2]), max3f(mx[3], mx[4], mx[5]), fmaxf(mx[6], mx[7])) * sc;
      // base-2 online softmax; the max is refreshed only when it grows by > 8
      const float mnew = fmaxf(m, mt);
      const bool resc = mnew > m + 8.f;
      const float factor = resc ? ex2(m - mnew) : 1.f;
      if (resc) m = mnew;
      const uint64_t NM2 = rowmask ? pk2(-INFINITY, -INFINITY) : pk2(-m, -m);
      uint64_t acc[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        uint32_t pk[32];
#pragma unroll
        for (int e = 0; e < 32; ++e) {
          const int c = 64 * half + 2 * e;
          const uint64_t t = ffma2(pk2(__uint_as_float(sr[c]), __uint_as_float(sr[c + 1])), SC2, NM2);
          float t0, t1;
          upk2(t, t0, t1);
          const float p0 = ex2(t0), p1 = ex2(t1);
          acc[e & 3] = fadd2(acc[e & 3], pk2(p0, p1));
          pk[e] = pack_bf16x2(p0, p1);
        }
        tmem_st32(tS + 32u * half, pk);
      }
      float s0, s1;
      upk2(fadd2(fadd2(acc[0], acc[1]), fadd2(acc[2], acc[3])), s0, s1);
      l = l * factor + (s0 + s1);
      if (__any_sync(0xffffffffu, resc && j > 0)) {
        // PV of the previous tile has retired (it precedes this tile's S commit)
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          uint32_t o[32];
          tmem_ld32(tO + 32u * c, o);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * factor);
          tmem_st32(tO + 32u * c, o);
        }
      }
      // the next tile's QK^T is issued only after this tile's P is ready, and this
      // tile's QK^T has retired: the query-side bias operand can be rewritten here
      if (s_next >= 0) {
        uint32_t w[8];
        aug_query_row(gauss ? none : nxt, xc, yc, inv_sc, w);
        store_aug_row(aq, r, w);
        fence_async_smem();
        aug_frame = s_next;
        cur = nxt;
      }
      tmem_wait_st();
      tc_fence_before();
      mbar_arrive(bar(B_PREADY(x)));
    }
    // ------------------------------------------------------------ epilogue
    const int64_t obase = (int64_t)layer * a.o_sl + (int64_t)p * a.o_st + (int64_t)head * a.o_sh;
    uint16_t* orow = static_cast<uint16_t*>(a.o) + obase;
    if (nt > 0 && ok) {
      if (!mbar_wait(bar(B_OFINAL(x)), 0, abort_flag, T)) { fail(P, abort_flag, 8); ok = false; }
    }
    ok = __all_sync(0xffffffffu, ok);
    const float inv = (l > 0.f) ? 1.f / l : 0.f;
    if (nt > 0 && ok) {
      tc_fence_after();
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        uint32_t o[32];
        tmem_ld32(tO + 32u * c, o);
        tmem_wait_ld();
        if (row_ok) {
          uint32_t w[16];
#pragma unroll
          for (int e = 0; e < 16; ++e)
            w[e] = pack_bf16x2(__uint_as_float(o[2 * e]) * inv, __uint_as_float(o[2 * e + 1]) * inv);
          uint4* dst = reinterpret_cast<uint4*>(orow + 32 * c);
#pragma unroll
          for (int e = 0; e < 4; ++e) dst[e] = make_uint4(w[4 * e], w[4 * e + 1], w[4 * e + 2], w[4 * e + 3]);
        }
      }
    } else if (row_ok) {
      uint4* dst = reinterpret_cast<uint4*>(orow);
      for (int e = 0; e < HD / 8; ++e) dst[e] = make_uint4(0, 0, 0, 0);
    }
    if (row_ok && a.lse)
      a.lse[((int64_t)layer * a.H + head) * a.Nq + p] = (l > 0.f) ? (m + log2f(l)) * 0.69314718055994531f : -INFINITY;
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kWarpMma) {
    __syncwarp();
    tmem_dealloc(tmem, TM_COLS);
  }
}

namespace {

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess)
    return nullptr;
  return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
}

// 4-D view [L][N][H][d] of a bf16 tensor; box = 64 elements of d x 1 head x 128 tokens.
bool make_map(PFN_cuTensorMapEncodeTiled_v12000 enc, CUtensorMap* m, const void* base, int64_t N, int64_t H,
              int64_t L, int64_t sl, int64_t st, int64_t sh) {
  cuuint64_t dims[4] = {(cuuint64_t)HD, (cuuint64_t)H, (cuuint64_t)N, (cuuint64_t)L};
  cuuint64_t strides[3] = {(cuuint64_t)(sh * 2), (cuuint64_t)(st * 2), (cuuint64_t)(sl * 2)};
  cuuint32_t box[4] = {64, 1, (cuuint32_t)BM, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

double bias_expansion_bound(float lambda, float sigma, int h, int w) {
  // the key operand holds x', y' (half-integers up to (w-1)/2) and q = x'^2 + y'^2 (two
  // terms) exactly in bf16 only while 2|x'|, 2|y'| < 256 and 4q < 2^16
  if (w > 256 || h > 256 || (int64_t)(w - 1) * (w - 1) + (int64_t)(h - 1) * (h - 1) >= 65536) return INFINITY;
  const double C = (double)lambda * 1.4426950408889634 / (2.0 * (double)sigma * (double)sigma);
  return C * ((double)w * w + (double)h * h) * 0x1p-24;
}

// The kernel's limits: bf16, d = 128, at most kMaxTiles KV tiles (each segment cut
// from its start, a retrieved one per frame; the largest segment lengths count),
// S <= 127 source frames, h w <= 65535, 16-byte aligned tensors and strides, sm_103.
bool attn_tc_supported(const AttnArgs& a) {
  if (a.dtype != CRC_BF16 || a.d != HD) return false;
  int64_t ntiles = 0;
  for (int g = 0; g < a.nseg; ++g) {
    const crc_segment& sg = a.seg[g];
    if (sg.length <= 0) continue;
    if (sg.kind == CRC_SEG_RETRIEVED || (sg.kind == CRC_SEG_CURRENT && a.frame_causal))
      ntiles += (int64_t)a.F * ((a.h * a.w + BN - 1) / BN);
    else
      ntiles += (sg.length + BN - 1) / BN;
  }
  if (ntiles > kMaxTiles || a.S > 127 || a.h * a.w > 65535) return false;
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  if (!al16(a.q) || !al16(a.k) || !al16(a.v) || !al16(a.o)) return false;
  const int64_t strides[9] = {a.q_sl, a.q_st, a.q_sh, a.k_sl, a.k_st, a.k_sh, a.o_sl, a.o_st, a.o_sh};
  for (int64_t x : strides)
    if ((x * 2) % 16 != 0) return false;
  int dev = 0, major = 0, minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  return major == 10 && minor == 3;
}

cudaError_t launch_attn_tc(const AttnArgs& a, cudaStream_t s) {
  if (!attn_tc_supported(a)) return cudaErrorNotSupported;
  auto enc = tensor_map_encoder();
  if (!enc) return cudaErrorNotSupported;
  CUtensorMap mq, mk, mv;
  if (!make_map(enc, &mq, a.q, a.Nq, a.H, a.L, a.q_sl, a.q_st, a.q_sh) ||
      !make_map(enc, &mk, a.k, a.Nk, a.H, a.L, a.k_sl, a.k_st, a.k_sh) ||
      !make_map(enc, &mv, a.v, a.Nk, a.H, a.L, a.k_sl, a.k_st, a.k_sh))
    return cudaErrorNotSupported;
  TcParams P;
  memset(&P, 0, sizeof(P));
  P.a = a;
  P.scale_log2 = (float)(1.4426950408889634 / sqrt((double)a.d));
  P.coef_log2 = (float)(-(double)a.lambda * 1.4426950408889634 / (2.0 * (double)a.sigma * (double)a.sigma));
  P.gauss_gc = (float)((double)a.lambda * sqrt((double)a.d));
  P.gauss_k = (float)(1.4426950408889634 / (2.0 * (double)a.sigma * (double)a.sigma));
  P.timeout_ns = 2000000000ull;
  const int mode = a.bias_form == 1 ? kBiasGauss
                   : (a.bias_direct || bias_expansion_bound(a.lambda, a.sigma, a.h, a.w) > kExpansionLimit)
                       ? kBiasDirect
                       : kBiasTensor;
  using KernelFn = void (*)(const CUtensorMap, const CUtensorMap, const CUtensorMap, const TcParams);
  static const KernelFn kernels[3][2] = {
      {attn_tc_kernel<kBiasTensor, false>, attn_tc_kernel<kBiasTensor, true>},
      {attn_tc_kernel<kBiasGauss, false>, attn_tc_kernel<kBiasGauss, true>},
      {attn_tc_kernel<kBiasDirect, false>, attn_tc_kernel<kBiasDirect, true>}};
  const KernelFn kernel = kernels[mode][a.frame_causal ? 1 : 0];
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
  if (e != cudaSuccess) return e;
  dim3 grid((a.Nq + NQT * BM - 1) / (NQT * BM), a.H, a.L);
  kernel<<<grid, kThreads, SMEM_BYTES, s>>>(mq, mk, mv, P);
  return cudaGetLastError();
}

}  // namespace crc
