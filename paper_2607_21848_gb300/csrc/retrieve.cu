// Loop-closure retrieval and gather (Sec. 4.2, Eq. 1), fused into one launch.
//
// Every CTA scores the whole bank in fp64 (no FMA contraction, fixed operation
// order), selects the k admissible chunks with the smallest (s(j), j) by k rounds
// of a block-wide lexicographic arg-min, applies the empty-set fallback (the slot
// extends the recent window), and then copies its share of the retrieved chunks'
// K/V rows from the slab pool into the retrieved cache segments.  CTA 0 also
// writes the indices, scores and count.  Recomputing the top-k in every CTA costs
// a few microseconds of ALU work on at most a few thousand entries and removes a
// launch and a grid-wide dependency from the chunk step.
#include <float.h>
#include <limits.h>

#include "gather.cuh"
#include "internal.cuh"

namespace crc {

namespace {

struct Cand {
  double s;
  int j;
};

__device__ __forceinline__ bool cand_less(double s1, int j1, double s2, int j2) {
  return (s1 < s2) || (s1 == s2 && j1 < j2);
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

}  // namespace

template <bool ROPE>
__global__ void __launch_bounds__(256, ROPE ? 2 : 4) retrieve_gather_kernel(const __grid_constant__ RetrieveArgs a) {
  __shared__ double sh_cn[3], sh_vn[3];
  __shared__ double red_s[8];
  __shared__ int red_j[8];
  __shared__ GatherPlan plan;
  __shared__ double slot_score[CRC_MAX_K];
  __shared__ int sh_count;
  const int tid = threadIdx.x;
  const int lane = tid & 31, warp = tid >> 5;

  if (tid == 0) {
    double c[3], v[3];
    chunk_summary(&a.cur.rec[0][0], a.cur.F, c, v);
    for (int e = 0; e < 3; ++e) {
      sh_cn[e] = c[e];
      sh_vn[e] = v[e];
    }
    sh_count = 0;
  }
  __syncthreads();
  double cn[3] = {sh_cn[0], sh_cn[1], sh_cn[2]};
  double vn[3] = {sh_vn[0], sh_vn[1], sh_vn[2]};

  // k rounds: round r finds the smallest admissible (s, j) strictly after round r-1's
  double ps = -DBL_MAX;
  int pj = INT_MIN;
  bool first = true;
  int count = 0;
  for (int r = 0; r < a.k; ++r) {
    double bs = __longlong_as_double(0x7ff0000000000000LL);  // +inf
    int bj = INT_MAX;
    for (int j = tid; j < a.count; j += blockDim.x) {
      double s, dist, dot;
      score_entry(a.centre, a.view, j, cn, vn, a.E, a.w_v, s, dist, dot);
      const bool adm = (dist <= a.tau_c) && (dot >= a.cos_tau_v) && (a.n - j >= a.delta) &&
                       !(a.exclude_sink && j == 0);
      const bool after = first || cand_less(ps, pj, s, j);
      if (adm && after && cand_less(s, j, bs, bj)) {
        bs = s;
        bj = j;
      }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const double os = __shfl_xor_sync(0xffffffffu, bs, o);
      const int oj = __shfl_xor_sync(0xffffffffu, bj, o);
      if (cand_less(os, oj, bs, bj)) {
        bs = os;
        bj = oj;
      }
    }
    if (lane == 0) {
      red_s[warp] = bs;
      red_j[warp] = bj;
    }
    __syncthreads();
    bs = red_s[0];
    bj = red_j[0];
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w)
      if (cand_less(red_s[w], red_j[w], bs, bj)) {
        bs = red_s[w];
        bj = red_j[w];
      }
    __syncthreads();
    if (bj == INT_MAX) break;  // block-uniform
    if (tid == 0) {
      plan.chunk[r] = bj;
      slot_score[r] = bs;
    }
    ps = bs;
    pj = bj;
    first = false;
    ++count;
  }
  if (tid == 0) {
    for (int r = count; r < a.k; ++r) {
      const int e = a.ext_first - (r - count);
      plan.chunk[r] = (a.ext_first >= 0 && e >= a.ext_min) ? e : -1;
      slot_score[r] = __longlong_as_double(0x7ff0000000000000LL);  // +inf
    }
    sh_count = count;
    if (blockIdx.x == 0) {
      for (int r = 0; r < a.k; ++r) {
        a.d_idx[r] = plan.chunk[r];
        if (a.d_score) a.d_score[r] = slot_score[r];
      }
      *a.d_count = count;
    }
  }
  __syncthreads();
  if (a.g.pool == nullptr) return;
  if (ROPE) plan_rope(a.g, a.k, plan);
  gather_slots<ROPE>(a.g, a.k, plan);
}

// The gather alone, for a cache that mirrors the retrieved slots of a step.
template <bool ROPE>
__global__ void __launch_bounds__(256, ROPE ? 2 : 4) gather_kernel(const __grid_constant__ GatherOnlyArgs a) {
  __shared__ GatherPlan plan;
  if (threadIdx.x < a.k) plan.chunk[threadIdx.x] = a.d_idx[threadIdx.x];
  __syncthreads();
  if (ROPE) plan_rope(a.g, a.k, plan);
  gather_slots<ROPE>(a.g, a.k, plan);
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

cudaError_t launch_retrieve(const RetrieveArgs& a, cudaStream_t s) {
  const int blocks = a.g.pool ? gather_blocks(a.k, a.g) : 1;
  if (a.g.pool && a.g.rope_pairs > 0)
    retrieve_gather_kernel<true><<<blocks, 256, 0, s>>>(a);
  else
    retrieve_gather_kernel<false><<<blocks, 256, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_gather(const GatherOnlyArgs& a, cudaStream_t s) {
  if (a.g.rope_pairs > 0)
    gather_kernel<true><<<gather_blocks(a.k, a.g), 256, 0, s>>>(a);
  else
    gather_kernel<false><<<gather_blocks(a.k, a.g), 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace crc
