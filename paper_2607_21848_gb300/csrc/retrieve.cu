// Loop-closure retrieval (Sec. 4.2, Eq. 1) and the gather of the retrieved chunks.
//
// Two launches.  The top-k launch scores every bank entry exactly once across its
// grid, in fp64 round-to-nearest without FMA contraction and in a fixed operation
// order, so that every score is bit-identical to a plain fp64 evaluation of Eq. 1.
// Each thread keeps the eight smallest admissible (s(j), j) of its entries; a block
// reduces its threads' lists to its k smallest.  With one block those are the
// result.  With several, every block writes its k candidates to the workspace and
// the last block to finish merges all of them.  The block that holds the result
// applies the empty-set fallback (the slot extends the recent window) and writes the
// indices, scores and count.  Selection is by the exact lexicographic order of
// (s(j), j), so the result does not depend on how entries are split over threads.
//
// The gather launch (a programmatic dependent launch: it is scheduled while the
// top-k grid runs and waits for its results before reading them) copies the
// retrieved chunks' K/V from the slab pool into the retrieved cache segments.
#include <limits.h>

#include "gather.cuh"
#include "internal.cuh"

namespace crc {

namespace {

constexpr int kTopkThreads = 256;
constexpr int kEntriesPerBlock = 512;  // bank entries per top-k block before the grid stops growing
constexpr int kMaxTopkBlocks = 2048;
constexpr int kList = 8;               // per-thread list length (>= CRC_MAX_K)
static_assert(kList >= CRC_MAX_K, "per-thread list shorter than k");

constexpr unsigned long long kNoKey = ~0ull;  // sentinel: no candidate

// fp64 score -> 64-bit key with the same order (no NaN reaches this: a NaN score
// fails the admissibility gates); -0 is folded onto +0 so that equal scores tie.
__device__ __forceinline__ unsigned long long score_key(double s) {
  if (s == 0.0) s = 0.0;
  const unsigned long long u = (unsigned long long)__double_as_longlong(s);
  return (u >> 63) ? ~u : (u | 0x8000000000000000ull);
}
__device__ __forceinline__ double key_score(unsigned long long k) {
  const unsigned long long u = (k >> 63) ? (k & 0x7fffffffffffffffull) : ~k;
  return __longlong_as_double((long long)u);
}

__device__ __forceinline__ bool cand_less(unsigned long long k1, int j1, unsigned long long k2, int j2) {
  return (k1 < k2) || (k1 == k2 && j1 < j2);
}

// Eq. 1 terms for bank entry j, fp64 round-to-nearest without contraction.
__device__ __forceinline__ void score_entry(const double* __restrict__ centre, const double* __restrict__ view, int j,
                                            const double cn[3], const double vn[3], double E, double w_v,
                                            double& s, double& dist, double& dot) {
  const double dx = __dsub_rn(centre[3 * j + 0], cn[0]);
  const double dy = __dsub_rn(centre[3 * j + 1], cn[1]);
  const double dz = __dsub_rn(centre[3 * j + 2], cn[2]);
  const double d2 = __dadd_rn(__dadd_rn(__dmul_rn(dx, dx), __dmul_rn(dy, dy)), __dmul_rn(dz, dz));
  dist = __ddiv_rn(__dsqrt_rn(d2), E);
  dot = __dadd_rn(__dadd_rn(__dmul_rn(view[3 * j + 0], vn[0]), __dmul_rn(view[3 * j + 1], vn[1])),
                  __dmul_rn(view[3 * j + 2], vn[2]));
  s = __dadd_rn(dist, __dmul_rn(w_v, __dsub_rn(1.0, dot)));
}

// A sorted list of the kList smallest candidates seen by one thread, in registers
// (every index below is a compile-time constant after unrolling).
struct List {
  unsigned long long key[kList];
  int j[kList];

  __device__ __forceinline__ void clear() {
#pragma unroll
    for (int i = 0; i < kList; ++i) {
      key[i] = kNoKey;
      j[i] = INT_MAX;
    }
  }
  __device__ __forceinline__ void insert(unsigned long long ck, int cj) {
    if (!cand_less(ck, cj, key[kList - 1], j[kList - 1])) return;
    key[kList - 1] = ck;
    j[kList - 1] = cj;
#pragma unroll
    for (int i = kList - 1; i > 0; --i) {
      if (cand_less(key[i], j[i], key[i - 1], j[i - 1])) {
        const unsigned long long tk = key[i];
        key[i] = key[i - 1];
        key[i - 1] = tk;
        const int tj = j[i];
        j[i] = j[i - 1];
        j[i - 1] = tj;
      }
    }
  }
  __device__ __forceinline__ void pop() {
#pragma unroll
    for (int i = 0; i < kList - 1; ++i) {
      key[i] = key[i + 1];
      j[i] = j[i + 1];
    }
    key[kList - 1] = kNoKey;
    j[kList - 1] = INT_MAX;
  }
};

struct BlockScratch {
  unsigned long long wkey[kTopkThreads / 32];
  int wj[kTopkThreads / 32];
  unsigned long long best_key;
  int best_j;
  int last;
};

// The k smallest candidates over the block's thread lists, into out_key/out_j
// (sentinels where fewer exist).  Every thread takes part; ends with a barrier.
__device__ void block_select(List& L, int k, BlockScratch& sh, unsigned long long* out_key, int* out_j) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int r = 0; r < k; ++r) {
    unsigned long long bk = L.key[0];
    int bj = L.j[0];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long ok = __shfl_xor_sync(0xffffffffu, bk, o);
      const int oj = __shfl_xor_sync(0xffffffffu, bj, o);
      if (cand_less(ok, oj, bk, bj)) {
        bk = ok;
        bj = oj;
      }
    }
    if (lane == 0) {
      sh.wkey[warp] = bk;
      sh.wj[warp] = bj;
    }
    __syncthreads();
    if (tid == 0) {
      unsigned long long mk = sh.wkey[0];
      int mj = sh.wj[0];
      for (int w = 1; w < kTopkThreads / 32; ++w)
        if (cand_less(sh.wkey[w], sh.wj[w], mk, mj)) {
          mk = sh.wkey[w];
          mj = sh.wj[w];
        }
      sh.best_key = mk;
      sh.best_j = mj;
      out_key[r] = mk;
      out_j[r] = mj;
    }
    __syncthreads();
    // j identifies one entry of the bank, so exactly one thread holds the winner
    if (sh.best_j != INT_MAX && L.j[0] == sh.best_j && L.key[0] == sh.best_key) L.pop();
  }
  __syncthreads();
}

}  // namespace

__global__ void __launch_bounds__(kTopkThreads) retrieve_topk_kernel(const __grid_constant__ RetrieveArgs a) {
  __shared__ double sh_cn[3], sh_vn[3];
  __shared__ BlockScratch sh;
  __shared__ unsigned long long res_key[CRC_MAX_K];
  __shared__ int res_j[CRC_MAX_K];
  const int tid = threadIdx.x;
  // let the gather grid begin its launch; it waits for this grid's results
  asm volatile("griddepcontrol.launch_dependents;");
  // the current chunk, the bank entries and the fallback: the arguments', or a step descriptor's
  int n = a.n, count = a.count, ext_first = a.ext_first;
  const double* cur = &a.cur.rec[0][0];
  if (a.step) {
    n = a.step->n;
    if (n < 0 || n >= a.capacity) {  // every block sees the same descriptor
      if (blockIdx.x == 0 && tid == 0) {
        atomicExch(a.status, CRC_STEP_BAD_DESCRIPTOR);
        for (int r = 0; r < a.k; ++r) {
          a.d_idx[r] = -1;
          if (a.d_score) a.d_score[r] = __longlong_as_double(0x7ff0000000000000LL);
        }
        *a.d_count = 0;
      }
      return;
    }
    count = n + 1;
    ext_first = a.step->ext_first;
    cur = reinterpret_cast<const double*>(a.step->frames);
  }
  if (tid == 0) {
    double c[3], v[3];
    chunk_summary(cur, a.cur.F, c, v);
    for (int e = 0; e < 3; ++e) {
      sh_cn[e] = c[e];
      sh_vn[e] = v[e];
    }
  }
  __syncthreads();
  const double cn[3] = {sh_cn[0], sh_cn[1], sh_cn[2]};
  const double vn[3] = {sh_vn[0], sh_vn[1], sh_vn[2]};

  List L;
  L.clear();
  const int stride = gridDim.x * blockDim.x;
  for (int j = blockIdx.x * blockDim.x + tid; j < count; j += stride) {
    double s, dist, dot;
    score_entry(a.centre, a.view, j, cn, vn, a.E, a.w_v, s, dist, dot);
    bool adm = (dist <= a.tau_c) && (dot >= a.cos_tau_v) && (n - j >= a.delta) && !(a.exclude_sink && j == 0);
    if (adm && a.slab_chunk) adm = a.slab_chunk[j % a.num_slabs] == j;  // its K/V slab still holds it
    if (adm) L.insert(score_key(s), j);
  }
  block_select(L, a.k, sh, res_key, res_j);

  if (gridDim.x > 1) {
    // hand the block's candidates to the last block to finish
    if (tid < a.k) {
      TopkCand c;
      c.key = res_key[tid];
      c.j = res_j[tid];
      c.pad = 0;
      a.partial[(size_t)blockIdx.x * a.k + tid] = c;
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) sh.last = atomicAdd(a.ticket, 1u) == gridDim.x - 1;
    __syncthreads();
    if (!sh.last) return;
    __threadfence();
    L.clear();
    const int n = gridDim.x * a.k;
    for (int i = tid; i < n; i += blockDim.x)  // other blocks' writes: read them from L2
      L.insert(__ldcg(&a.partial[i].key), __ldcg(&a.partial[i].j));
    block_select(L, a.k, sh, res_key, res_j);
  }

  if (tid == 0) {
    int found = 0;
    while (found < a.k && res_j[found] != INT_MAX) ++found;
    const int count = found;
    for (int r = 0; r < a.k; ++r) {
      int chunk;
      double score;
      if (r < count) {
        chunk = res_j[r];
        score = key_score(res_key[r]);
      } else {
        // the slot extends the recent window with the next-older chunk, if it is kept
        const int e = ext_first - (r - count);
        const bool ok = ext_first >= 0 && e >= a.ext_min && e >= 0 &&
                        (a.slab_chunk == nullptr || a.slab_chunk[e % a.num_slabs] == e);
        chunk = ok ? e : -1;
        score = __longlong_as_double(0x7ff0000000000000LL);  // +inf
      }
      a.d_idx[r] = chunk;
      if (a.d_score) a.d_score[r] = score;
    }
    *a.d_count = count;
  }
}

// The gather alone: every slot's chunk comes from d_idx.  After a top-k launch it is
// a programmatic dependent launch, and griddepcontrol.wait holds it until the top-k
// results are visible; launched on its own, the wait returns at once.
template <bool ROPE>
__global__ void __launch_bounds__(256, 4) gather_kernel(const __grid_constant__ GatherOnlyArgs a) {
  __shared__ GatherPlan plan;
  asm volatile("griddepcontrol.wait;" ::: "memory");
  if (threadIdx.x < a.k) plan.chunk[threadIdx.x] = a.d_idx[threadIdx.x];
  __syncthreads();
  if (ROPE) plan_rope(a.g, a.k, plan, a.g.step ? a.g.step->rope_pos_slot0 : a.g.rope_pos_slot0);
  gather_slots<ROPE>(a.g, a.k, plan);
}

int retrieve_blocks(int32_t count) {
  int64_t b = ((int64_t)count + kEntriesPerBlock - 1) / kEntriesPerBlock;
  if (b < 1) b = 1;
  if (b > kMaxTopkBlocks) b = kMaxTopkBlocks;
  return (int)b;
}

size_t retrieve_workspace_bytes(int32_t count, int32_t k) {
  const int b = retrieve_blocks(count);
  if (b <= 1) return 0;
  const size_t cands = ((size_t)b * k * sizeof(TopkCand) + 255) / 256 * 256;
  return cands + 256;  // + the ticket counter
}

namespace {

// One warp per row; at most four CTAs of 256 threads per SM, grid-stride beyond that.
int gather_blocks(int k, const GatherArgs& g) {
  const int64_t rows = 2LL * k * g.L * g.Nc;
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (rows + 7) / 8;
  int blocks = (int)(want < (int64_t)sms * 4 ? want : (int64_t)sms * 4);
  return blocks < 1 ? 1 : blocks;
}

}  // namespace

cudaError_t launch_retrieve(const RetrieveArgs& a, const GatherArgs& g, cudaStream_t s) {
  const int blocks = retrieve_blocks(a.count);
  if (blocks > 1) {
    cudaError_t e = cudaMemsetAsync(a.ticket, 0, sizeof(unsigned int), s);
    if (e != cudaSuccess) return e;
  }
  retrieve_topk_kernel<<<blocks, kTopkThreads, 0, s>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || g.pool == nullptr) return e;
  GatherOnlyArgs ga;
  ga.d_idx = a.d_idx;
  ga.k = a.k;
  ga.g = g;
  return launch_gather(ga, s, true);
}

cudaError_t launch_gather(const GatherOnlyArgs& a, cudaStream_t s, bool after_topk) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(gather_blocks(a.k, a.g));
  cfg.blockDim = dim3(256);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = after_topk ? 1 : 0;
  if (a.g.rope_pairs > 0) return cudaLaunchKernelEx(&cfg, gather_kernel<true>, a);
  return cudaLaunchKernelEx(&cfg, gather_kernel<false>, a);
}

}  // namespace crc
