// rules.cu -- the selection rules of the paper's component ablation, beside
// the register-anchored threshold of the method (Eqs. 5 and 8):
//   mean_ref_kernel     the "mean threshold" reference: per segment or per
//                       sample, the mean score of the unit's candidate rows
//                       (visual rows, restricted to a previous keep mask);
//                       the threshold is then s(v) >= lambda * mean;
//   budget_keep_kernel  the "fixed budget" rule, i.e. the top-K rule of
//                       Sec. 2, S = top-K(V, s): per sample the budget[b]
//                       candidate rows with the largest score, equal scores
//                       taken lower row first.
//   pool_scores_kernel  scores of merged tokens from their patches' scores
//                       (a 2x2 patch merger puts a merged token's patches on
//                       consecutive rows): the sum, mean or max of each
//                       group of consecutive rows.
// All are deterministic: fixed-order sums, and a selection whose result
// does not depend on thread timing.
#include "common.cuh"
#include "kernels.cuh"

namespace occam {

__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// One CTA of 256 threads per unit (segment or sample). Thread t sums the
// candidate rows t, t + 256, ... in fp64; warps then combine in a fixed tree
// and warp 0's lane 0 adds the eight warp sums in order.
__global__ void __launch_bounds__(256) mean_ref_kernel(MeanRefParams p) {
  __shared__ double wsum[8];
  __shared__ int wcnt[8];
  const int u = blockIdx.x, tid = threadIdx.x;
  const int64_t lo = p.scope == OCCAM_REF_SEGMENT ? p.bt.seg_off[u] : p.bt.row_off[u];
  const int64_t hi = p.scope == OCCAM_REF_SEGMENT ? p.bt.seg_off[u + 1] : p.bt.row_off[u + 1];
  double acc = 0.0;
  int cnt = 0;
  for (int64_t r = lo + tid; r < hi; r += blockDim.x) {
    if (p.role[r] == 0 && (!p.prev_keep || p.prev_keep[r] != 0)) {
      acc += (double)p.s[r];
      ++cnt;
    }
  }
  acc = warp_sum_d(acc);
  cnt = warp_sum_i(cnt);
  if ((tid & 31) == 0) {
    wsum[tid >> 5] = acc;
    wcnt[tid >> 5] = cnt;
  }
  __syncthreads();
  if (tid == 0) {
    double a = 0.0;
    int c = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
      a += wsum[w];
      c += wcnt[w];
    }
    const float ref = c > 0 ? (float)(a / (double)c) : 0.f;
    p.ref[u] = ref;
    if (p.tau) p.tau[u] = p.lambda * ref;
  }
}

// Order-preserving 32-bit key of a float: larger values give larger keys
// (-0 is taken as +0, so equal values have equal keys; NaN is undefined).
__device__ __forceinline__ uint32_t order_key(float v) {
  const uint32_t u = __float_as_uint(v == 0.f ? 0.f : v);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// One CTA of 1,024 threads per sample.
//   1. n = the sample's candidate count; K = clamp(budget[b], 0, n).
//   2. If 0 < K < n: the K-th largest candidate key t, most significant byte
//      first (per byte a 256-bin histogram of the keys that match the bytes
//      chosen so far, one histogram per warp, summed; then the bucket where
//      the running count from the top reaches K). need = how many keys equal
//      to t are kept = K - #(keys > t).
//   3. Each thread takes a contiguous run of the sample's rows: keys above t
//      are kept; keys equal to t are ranked in row order by a block scan and
//      the first `need` of them kept. Register rows get keep_registers.
__global__ void __launch_bounds__(1024) budget_keep_kernel(BudgetParams p) {
  __shared__ uint32_t hist[32][256];
  __shared__ uint32_t tot[256];
  __shared__ uint32_t s_prefix, s_k;
  __shared__ int s_cnt;
  __shared__ int tmp[40];
  const int b = blockIdx.x, tid = threadIdx.x, warp = tid >> 5;
  const int64_t lo = p.bt.row_off[b], hi = p.bt.row_off[b + 1];
  auto cand = [&](int64_t r) { return p.role[r] == 0 && (!p.prev_keep || p.prev_keep[r] != 0); };
  if (tid == 0) s_cnt = 0;
  __syncthreads();
  int c = 0;
  for (int64_t r = lo + tid; r < hi; r += blockDim.x) c += cand(r) ? 1 : 0;
  c = warp_sum_i(c);
  if ((tid & 31) == 0) atomicAdd(&s_cnt, c);
  __syncthreads();
  const int n = s_cnt;
  const int K = min(max(p.budget[b], 0), n);
  // t = 0 with need = n keeps every candidate (every key is >= 0)
  uint32_t t = 0;
  int need = n;
  if (K == 0) {
    t = 0xffffffffu;
    need = 0;
  } else if (K < n) {
    if (tid == 0) {
      s_prefix = 0;
      s_k = (uint32_t)K;
    }
    uint32_t mask = 0;
    for (int shift = 24; shift >= 0; shift -= 8) {
      for (int i = tid; i < 32 * 256; i += blockDim.x) (&hist[0][0])[i] = 0;
      __syncthreads();
      const uint32_t prefix = s_prefix;
      for (int64_t r = lo + tid; r < hi; r += blockDim.x) {
        if (!cand(r)) continue;
        const uint32_t key = order_key(p.s[r]);
        if ((key & mask) == prefix) atomicAdd(&hist[warp][(key >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (tid < 256) {
        uint32_t s = 0;
        for (int w = 0; w < 32; ++w) s += hist[w][tid];
        tot[tid] = s;
      }
      __syncthreads();
      if (tid == 0) {
        uint32_t k = s_k, cum = 0;
        int d = 255;
        for (; d > 0; --d) {
          if (cum + tot[d] >= k) break;
          cum += tot[d];
        }
        s_k = k - cum;
        s_prefix = prefix | ((uint32_t)d << shift);
      }
      mask |= 255u << shift;
      __syncthreads();
    }
    t = s_prefix;
    need = (int)s_k;
  }
  // contiguous runs of rows per thread keep the tie ranking in row order
  const int64_t nrows = hi - lo;
  const int64_t per = (nrows + blockDim.x - 1) / blockDim.x;
  const int64_t a = lo + min(nrows, (int64_t)tid * per), z = lo + min(nrows, ((int64_t)tid + 1) * per);
  int ties = 0;
  for (int64_t r = a; r < z; ++r)
    if (cand(r) && order_key(p.s[r]) == t) ++ties;
  int ties_total;
  int rank = block_exclusive_scan(ties, tmp, &ties_total);
  for (int64_t r = a; r < z; ++r) {
    bool k;
    if (p.role[r] != 0) {
      k = p.keep_registers != 0;
    } else if (!cand(r)) {
      k = false;
    } else {
      const uint32_t key = order_key(p.s[r]);
      if (key == t) {
        k = rank < need;
        ++rank;
      } else {
        k = key > t;
      }
    }
    p.keep[r] = k ? 1 : 0;
  }
  if (tid == 0 && p.count_vis) p.count_vis[b] = K;
}

// One thread per merged row; the group's values are added in row order.
__global__ void __launch_bounds__(256) pool_scores_kernel(const float* __restrict__ s_in, int64_t rows_out, int group,
                                                          int mode, float* __restrict__ s_out) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < rows_out; i += (int64_t)gridDim.x * blockDim.x) {
    const float* g = s_in + i * group;
    float acc = g[0];
    for (int k = 1; k < group; ++k) acc = mode == OCCAM_POOL_MAX ? fmaxf(acc, g[k]) : acc + g[k];
    s_out[i] = mode == OCCAM_POOL_MEAN ? acc / (float)group : acc;
  }
}

}  // namespace occam
