// Biased flash attention on the 5th-generation tensor cores (Sec. 4.3, Eq. 2).
//
//   A_pk = q_p . k_k / sqrt(d) + lambda B_s(p, k),  B = -||u_k - u^_s(p)||^2 / (2 sigma^2)
//
// on retrieved-slot key columns with a valid correspondence, 0 elsewhere; the
// bias is evaluated per (query row, key column) inside the tile loop and never
// written anywhere.  bf16 Q/K/V, fp32 scores, softmax and accumulation, bf16 O.
//
// Structure (one CTA = two 128-row query tiles of one (layer, head)):
//   warps 0-3  softmax of query tile 0   (TMEM lanes 0-127 of S0/O0)
//   warps 4-7  softmax of query tile 1   (TMEM lanes 0-127 of S1/O1)
//   warp  8    TMA producer: Q once, then K/V tiles of 128 keys, 2 stages each,
//              128-byte swizzled boxes of 128 rows x 64 elements
//   warp  9    TMEM owner and single-thread tcgen05.mma issuer
//   warps 10-11 idle (they complete the third warpgroup for the register split)
// TMEM (512 columns): S0 | S1 | O0 | O1, 128 fp32 columns each.  S = Q K^T is an
// SS MMA (both operands K-major in shared memory); each softmax thread reads its
// row of S, writes P in bf16 over the first 64 columns of the same S buffer and
// the MMA warp accumulates O += P V with P taken straight from TMEM (TS MMA, V
// MN-major in shared memory).  The MMA warp alternates the two query tiles, so
// the tensor core works on one tile while the other tile's softmax runs.
// Online softmax in base 2 with the row max kept stale until it grows by more
// than 2^8 (exact: the same max normalises P, O and the row sum); O in TMEM is
// rescaled only on those rare steps.  KV tiles that hold no active key (an empty
// retrieved slot, keys past the cache end) are skipped by every role.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <math.h>
#include <string.h>

#include "internal.cuh"
#include "keys.cuh"
#include "tc_ptx.cuh"

namespace crc {

namespace {

using namespace ptx;

constexpr int BM = 128;  // query rows per tile = TMEM lanes
constexpr int BN = 128;  // keys per KV tile
constexpr int HD = 128;  // head dim
constexpr int NQT = 2;   // query tiles per CTA
constexpr int ST = 2;    // stages for K and for V
constexpr int kThreads = 384;  // 3 warpgroups: softmax 0, softmax 1, producer/MMA
constexpr int kWarpTma = 8;
constexpr int kWarpMma = 9;
// register split (setmaxnreg): the block launches with 384 x 168 registers; the
// producer warpgroup drops to 96 and each softmax warpgroup rises to 200:
// 2 x 128 x 200 + 128 x 96 <= 384 x 168.
constexpr int kRegsSoftmax = 200;
constexpr int kRegsProducer = 96;
static_assert(2 * 128 * kRegsSoftmax + 128 * kRegsProducer <= kThreads * 168, "register split exceeds the launch");
constexpr int BOX = BM * 64 * 2;  // 128 rows x 64 bf16 = 16 KB
constexpr int TILE = 2 * BOX;     // 128 rows x 128 bf16 = 32 KB
constexpr int kMaxTiles = 1024;   // KV tiles per call

constexpr int OFF_Q = 0;
constexpr int OFF_K = OFF_Q + NQT * TILE;
constexpr int OFF_V = OFF_K + ST * TILE;
constexpr int OFF_TAB = OFF_V + ST * TILE;
constexpr int TAB_BYTES = NQT * 2 * BN * 16;
constexpr int OFF_TILES = OFF_TAB + TAB_BYTES;
constexpr int OFF_BAR = OFF_TILES + kMaxTiles * 8;
constexpr int NBAR = 1 + 4 * ST + 3 * NQT + 1;
constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
constexpr int SMEM_BYTES = OFF_MISC + 64 + 1024;  // + slack for 1024-byte alignment

constexpr uint32_t TM_S = 0;    // S/P of tile x at column 128 x
constexpr uint32_t TM_O = 256;  // O of tile x at column 256 + 128 x
constexpr uint32_t TM_COLS = 512;

constexpr uint8_t CLS_PLAIN = 0;    // every column active, none biased
constexpr uint8_t CLS_BIAS1 = 1;    // every column active and biased, one source frame
constexpr uint8_t CLS_GENERAL = 2;  // anything else: per-column bias / mask

struct TileInfo {
  uint16_t tile;
  uint8_t cls;
  int8_t sA, sB;  // the (at most two) source frames of biased columns, -1 if none
  uint8_t pad[3];
};

struct TcParams {
  AttnArgs a;
  float scale_log2;  // log2(e) / sqrt(d)
  float coef_log2;   // -lambda log2(e) / (2 sigma^2)
  uint64_t timeout_ns;
};

// barrier indices
__device__ __forceinline__ int B_QFULL() { return 0; }
__device__ __forceinline__ int B_KFULL(int s) { return 1 + s; }
__device__ __forceinline__ int B_KEMPTY(int s) { return 1 + ST + s; }
__device__ __forceinline__ int B_VFULL(int s) { return 1 + 2 * ST + s; }
__device__ __forceinline__ int B_VEMPTY(int s) { return 1 + 3 * ST + s; }
__device__ __forceinline__ int B_SFULL(int x) { return 1 + 4 * ST + x; }
__device__ __forceinline__ int B_PREADY(int x) { return 1 + 4 * ST + NQT + x; }
__device__ __forceinline__ int B_OFINAL(int x) { return 1 + 4 * ST + 2 * NQT + x; }
__device__ __forceinline__ int B_DRAIN() { return 1 + 4 * ST + 3 * NQT; }

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
__device__ __forceinline__ uint64_t fsub2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ uint64_t fmul2(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ float max3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// One query row's correspondences in the two source frames of a KV tile, with the
// bias coefficient already zero for invalid pairs (exact fallback).
struct Corr {
  float uxA, uyA, cA, uxB, uyB, cB;
};

__device__ __forceinline__ Corr load_corr(const AttnArgs& a, const TileInfo* tiles, int j, int nt, int p, bool row_ok,
                                          float coef) {
  Corr c{0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  if (j >= nt || !row_ok) return c;
  const TileInfo ti = tiles[j];
  if (ti.sA < 0) return c;
  const int64_t ia = (int64_t)p * a.S + ti.sA, ib = (int64_t)p * a.S + ti.sB;
  const float2* uv = reinterpret_cast<const float2*>(a.uv);
  if (__ldg(a.valid + ia)) {
    const float2 u = __ldg(uv + ia);
    c.uxA = u.x;
    c.uyA = u.y;
    c.cA = coef;
  }
  if (__ldg(a.valid + ib)) {
    const float2 u = __ldg(uv + ib);
    c.uxB = u.x;
    c.uyB = u.y;
    c.cB = coef;
  }
  return c;
}

__device__ __forceinline__ void fail(const TcParams& P, volatile int* abort_flag, int code) {
  *abort_flag = 1;
  if (P.a.status) atomicExch(P.a.status, code);
}

}  // namespace

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

  if (tid == 0) {
    mbar_init(bar(B_QFULL()), 1);
    for (int s = 0; s < ST; ++s) {
      mbar_init(bar(B_KFULL(s)), 1);
      mbar_init(bar(B_KEMPTY(s)), 1);
      mbar_init(bar(B_VFULL(s)), 1);
      mbar_init(bar(B_VEMPTY(s)), 1);
    }
    for (int x = 0; x < NQT; ++x) {
      mbar_init(bar(B_SFULL(x)), 1);
      mbar_init(bar(B_PREADY(x)), BM);
      mbar_init(bar(B_OFINAL(x)), 1);
    }
    mbar_init(bar(B_DRAIN()), 1);
    *abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 0) {
    // compact list of KV tiles holding at least one active key, with their class
    const int ntot = (a.Nk + BN - 1) / BN;
    const int hw = a.h * a.w;
    int count = 0;
    for (int base = 0; base < ntot; base += 32) {
      const int t = base + lane;
      bool act = false;
      TileInfo ti;
      ti.tile = (uint16_t)t;
      ti.cls = CLS_GENERAL;
      ti.sA = -1;
      ti.sB = -1;
      if (t < ntot) {
        const int k0 = t * BN, k1 = k0 + BN;
        int nact = 0, nbias = 0, sA = 1 << 20, sB = -1;
        for (int g = 0; g < a.nseg; ++g) {
          const crc_segment sg = a.seg[g];
          if (sg.length <= 0) continue;
          const int lo = max(k0, sg.offset), hi = min(k1, sg.offset + sg.length);
          if (lo >= hi) continue;
          if (sg.kind == CRC_SEG_RETRIEVED) {
            if (a.slot_chunk && a.slot_chunk[sg.slot] < 0) continue;
            sA = min(sA, sg.slot * a.F + (lo - sg.offset) / hw);
            sB = max(sB, sg.slot * a.F + (hi - 1 - sg.offset) / hw);
            nbias += hi - lo;
          }
          nact += hi - lo;
        }
        act = nact > 0;
        if (sB >= 0) {
          ti.sA = (int8_t)sA;
          ti.sB = (int8_t)sB;
        }
        ti.cls = (nact == BN && sB < 0) ? CLS_PLAIN
                 : (nact == BN && nbias == BN && sA == sB) ? CLS_BIAS1 : CLS_GENERAL;
      }
      const unsigned m = __ballot_sync(0xffffffffu, act);
      if (act) tiles[count + __popc(m & ((1u << lane) - 1u))] = ti;
      count += __popc(m);
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
      int issued_k = 0, issued_v = 0;
      for (int j = 0; j < nt; ++j) {
        const int st = j % ST;
        const uint32_t par = ((j / ST) & 1) ^ 1;
        const int key0 = tiles[j].tile * BN;
        if (!mbar_wait(bar(B_KEMPTY(st)), par, abort_flag, T)) { fail(P, abort_flag, 1); break; }
        mbar_arrive_expect_tx(bar(B_KFULL(st)), TILE);
        for (int b = 0; b < 2; ++b)
          tma_load_4d(sbase + OFF_K + st * TILE + b * BOX, &tmK, bar(B_KFULL(st)), b * 64, head, key0, layer);
        issued_k = j + 1;
        if (!mbar_wait(bar(B_VEMPTY(st)), par, abort_flag, T)) { fail(P, abort_flag, 2); break; }
        mbar_arrive_expect_tx(bar(B_VFULL(st)), TILE);
        for (int b = 0; b < 2; ++b)
          tma_load_4d(sbase + OFF_V + st * TILE + b * BOX, &tmV, bar(B_VFULL(st)), b * 64, head, key0, layer);
        issued_v = j + 1;
      }
      if (*abort_flag) {
        // let the copies already issued land before the CTA can exit
        const uint64_t lim = 100000000ull;
        volatile int never = 0;
        mbar_wait(bar(B_QFULL()), 0, &never, lim);
        for (int j = (issued_k > ST ? issued_k - ST : 0); j < issued_k; ++j)
          mbar_wait(bar(B_KFULL(j % ST)), (j / ST) & 1, &never, lim);
        for (int j = (issued_v > ST ? issued_v - ST : 0); j < issued_v; ++j)
          mbar_wait(bar(B_VFULL(j % ST)), (j / ST) & 1, &never, lim);
      }
    }
   } else if (warp == kWarpMma) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0 && nt > 0) {
      constexpr uint32_t idesc_qk = idesc_bf16_f32(BM, BN, 0, 0);
      constexpr uint32_t idesc_pv = idesc_bf16_f32(BM, HD, 0, 1);
      // descriptors of the operand bases; advancing along K adds (bytes >> 4) to the
      // start-address field, which cannot carry out of its 14 bits for shared memory
      const uint64_t dq0 = sdesc_sw128(sbase + OFF_Q, 16, 1024);
      const uint64_t dk0 = sdesc_sw128(sbase + OFF_K, 16, 1024);
      const uint64_t dv0 = sdesc_sw128(sbase + OFF_V, BOX, 1024);
      auto issue_qk = [&](int x, int st) {
        const uint64_t ad = dq0 + (uint64_t)((x * TILE) >> 4);
        const uint64_t bd = dk0 + (uint64_t)((st * TILE) >> 4);
        const uint32_t d = tmem + TM_S + 128u * x;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const uint64_t off = (uint64_t)(((kk >> 2) * BOX + (kk & 3) * 32) >> 4);
          mma_ss(d, ad + off, bd + off, idesc_qk, kk > 0 ? 1u : 0u);
        }
      };
      auto issue_pv = [&](int x, int st, bool acc) {
        const uint64_t bd = dv0 + (uint64_t)((st * TILE) >> 4);
        const uint32_t d = tmem + TM_O + 128u * x;
        const uint32_t pa = tmem + TM_S + 128u * x;
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk)
          mma_ts(d, pa + 8u * kk, bd + (uint64_t)((kk * 2048) >> 4), idesc_pv, (acc || kk > 0) ? 1u : 0u);
      };
      bool ok = mbar_wait(bar(B_QFULL()), 0, abort_flag, T) && mbar_wait(bar(B_KFULL(0)), 0, abort_flag, T);
      if (!ok) fail(P, abort_flag, 3);
      if (ok) {
        tc_fence_after();
        issue_qk(0, 0);
        mma_commit(bar(B_SFULL(0)));
        issue_qk(1, 0);
        mma_commit(bar(B_SFULL(1)));
        mma_commit(bar(B_KEMPTY(0)));
        for (int j = 0; j < nt && ok; ++j) {
          const int st = j % ST;
          const int jn = j + 1, stn = jn % ST;
          const bool more = jn < nt;
          ok = mbar_wait(bar(B_PREADY(0)), j & 1, abort_flag, T) &&
               mbar_wait(bar(B_VFULL(st)), (j / ST) & 1, abort_flag, T);
          if (!ok) { fail(P, abort_flag, 4); break; }
          tc_fence_after();
          issue_pv(0, st, j > 0);
          if (more) {
            ok = mbar_wait(bar(B_KFULL(stn)), (jn / ST) & 1, abort_flag, T);
            if (!ok) { fail(P, abort_flag, 5); break; }
            tc_fence_after();
            issue_qk(0, stn);
            mma_commit(bar(B_SFULL(0)));
          } else {
            mma_commit(bar(B_OFINAL(0)));
          }
          ok = mbar_wait(bar(B_PREADY(1)), j & 1, abort_flag, T);
          if (!ok) { fail(P, abort_flag, 6); break; }
          tc_fence_after();
          issue_pv(1, st, j > 0);
          mma_commit(bar(B_VEMPTY(st)));
          if (more) {
            issue_qk(1, stn);
            mma_commit(bar(B_SFULL(1)));
            mma_commit(bar(B_KEMPTY(stn)));
          } else {
            mma_commit(bar(B_OFINAL(1)));
          }
        }
      }
      // every MMA issued so far has retired once this barrier fires
      volatile int never = 0;
      mma_commit(bar(B_DRAIN()));
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
    const int twg = tid - x * BM;     // thread index in the warpgroup
    const bool row_ok = p < a.Nq;
    const uint32_t trow = tmem + ((uint32_t)(wq * 32) << 16);
    const uint32_t tS = trow + TM_S + 128u * x;
    const uint32_t tO = trow + TM_O + 128u * x;
    float4* tab = reinterpret_cast<float4*>(smem + OFF_TAB) + x * 2 * BN;
    // scores stay in raw units z = q.k (+ bias / scale); one FMA per element maps
    // them to log2 units for the exponent: p = 2^(z * sc - m)
    const float sc = P.scale_log2;
    const float cb = P.coef_log2 / sc;
    const uint64_t SC2 = pk2(sc, sc);
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    // per-row correspondence of the (at most two) source frames of a tile,
    // loaded one tile ahead so that the global-load latency overlaps a tile
    Corr nxt = load_corr(a, tiles, 0, nt, p, row_ok, cb);
    for (int j = 0; j < nt; ++j) {
      const TileInfo ti = tiles[j];
      const Corr cur = nxt;
      nxt = load_corr(a, tiles, j + 1, nt, p, row_ok, cb);
      float4* tb = tab + (j & 1) * BN;
      if (ti.cls != CLS_PLAIN) {
        const KeyInfo ki = key_info_of(a, ti.tile * BN + twg);
        if (ti.cls == CLS_BIAS1) {
          reinterpret_cast<float2*>(tb)[twg] = make_float2(ki.x, ki.y);
        } else {
          const float sel = ki.src < 0 ? 0.f : (ki.src == ti.sA ? 1.f : 2.f);
          tb[twg] = make_float4(ki.x, ki.y, sel, ki.active ? 1.f : 0.f);
        }
        named_bar_sync(1 + x, BM);
      }
      if (ok && !mbar_wait(bar(B_SFULL(x)), j & 1, abort_flag, T)) { fail(P, abort_flag, 7); ok = false; }
      ok = __all_sync(0xffffffffu, ok);
      // after a failure keep walking the tile list: every warp of the group must
      // reach the same named barriers, so none of them can be left waiting
      if (!ok) continue;
      tc_fence_after();
      if (ti.cls == CLS_GENERAL) {
        // rare tiles (segment or frame boundaries, masked keys): per-column bias and
        // mask applied in place in TMEM, 32 columns at a time
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          uint32_t g[32];
          tmem_ld32(tS + 32u * c, g);
          tmem_wait_ld();
#pragma unroll
          for (int e = 0; e < 32; ++e) {
            const float4 t = tb[32 * c + e];
            const bool selB = t.z > 1.5f;
            const float ux = selB ? cur.uxB : cur.uxA, uy = selB ? cur.uyB : cur.uyA;
            const float cf = t.z > 0.5f ? (selB ? cur.cB : cur.cA) : 0.f;
            const float dx = t.x - ux, dy = t.y - uy;
            const float z = fmaf(cf, fmaf(dx, dx, dy * dy), __uint_as_float(g[e]));
            g[e] = __float_as_uint(t.w > 0.5f ? z : -INFINITY);
          }
          tmem_st32(tS + 32u * c, g);
        }
        tmem_wait_st();
      }
      uint32_t sr[128];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(tS + 32u * c, *reinterpret_cast<uint32_t(*)[32]>(&sr[32 * c]));
      tmem_wait_ld();
      if (ti.cls == CLS_BIAS1) {
        // all 128 keys in one source frame: z += cA ((x - ux)^2 + (y - uy)^2), two columns per op
        const uint64_t UX2 = pk2(cur.uxA, cur.uxA), UY2 = pk2(cur.uyA, cur.uyA), CA2 = pk2(cur.cA, cur.cA);
        const float4* t4 = tb;
#pragma unroll
        for (int c = 0; c < 128; c += 2) {
          const float4 t = t4[c >> 1];
          const uint64_t dx = fsub2(pk2(t.x, t.z), UX2);
          const uint64_t dy = fsub2(pk2(t.y, t.w), UY2);
          const uint64_t d2 = ffma2(dy, dy, fmul2(dx, dx));
          const uint64_t z = ffma2(d2, CA2, pk2(__uint_as_float(sr[c]), __uint_as_float(sr[c + 1])));
          float z0, z1;
          upk2(z, z0, z1);
          sr[c] = __float_as_uint(z0);
          sr[c + 1] = __float_as_uint(z1);
        }
      }
      // row max by a tree of three-input max operations
      float mx[43];
#pragma unroll
      for (int i = 0; i < 42; ++i)
        mx[i] = max3f(__uint_as_float(sr[3 * i]), __uint_as_float(sr[3 * i + 1]), __uint_as_float(sr[3 * i + 2]));
      mx[42] = fmaxf(__uint_as_float(sr[126]), __uint_as_float(sr[127]));
#pragma unroll
      for (int i = 0; i < 14; ++i) mx[i] = max3f(mx[3 * i], mx[3 * i + 1], mx[3 * i + 2]);
      mx[14] = mx[42];
#pragma unroll
      for (int i = 0; i < 5; ++i) mx[i] = max3f(mx[3 * i], mx[3 * i + 1], mx[3 * i + 2]);
      const float mt = max3f(max3f(mx[0], mx[1], mx[2]), mx[3], mx[4]) * sc;
      // base-2 online softmax; the max is refreshed only when it grows by > 8
      const float mnew = fmaxf(m, mt);
      const bool resc = mnew > m + 8.f;
      const float factor = resc ? ex2(m - mnew) : 1.f;
      if (resc) m = mnew;
      const uint64_t NM2 = pk2(-m, -m);
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
      float s0, s1, s2, s3;
      upk2(fadd2(fadd2(acc[0], acc[1]), fadd2(acc[2], acc[3])), s0, s1);
      (void)s2;
      (void)s3;
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

cudaError_t launch_attn_tc(const AttnArgs& a, cudaStream_t s) {
  if (a.dtype != CRC_BF16 || a.d != HD) return cudaErrorNotSupported;
  const int64_t ntiles = (a.Nk + BN - 1) / BN;
  if (ntiles > kMaxTiles || a.S > 127) return cudaErrorNotSupported;
  for (int g = 0; g < a.nseg; ++g)  // at most two source frames per KV tile
    if (a.seg[g].kind == CRC_SEG_RETRIEVED && a.seg[g].length > 0 && a.h * a.w < BN) return cudaErrorNotSupported;
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  if (!al16(a.q) || !al16(a.k) || !al16(a.v) || !al16(a.o)) return cudaErrorNotSupported;
  const int64_t strides[9] = {a.q_sl, a.q_st, a.q_sh, a.k_sl, a.k_st, a.k_sh, a.o_sl, a.o_st, a.o_sh};
  for (int64_t x : strides)
    if ((x * 2) % 16 != 0) return cudaErrorNotSupported;
  int dev = 0, major = 0, minor = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  if (major != 10 || minor != 3) return cudaErrorNotSupported;
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
  P.timeout_ns = 2000000000ull;
  cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
  if (e != cudaSuccess) return e;
  dim3 grid((a.Nq + NQT * BM - 1) / (NQT * BM), a.H, a.L);
  attn_tc_kernel<<<grid, kThreads, SMEM_BYTES, s>>>(mq, mk, mv, P);
  return cudaGetLastError();
}

}  // namespace crc
