// compact.cu -- order-preserving stream compaction of the kept rows and the
// gather of their hidden / K / V rows (Algorithm 1: decoding continues on
// [S2; T]; App. A, Eq. 21: the KV cache shrinks with the kept count).
//
// scan_kernel: single pass over the batch's row space in tiles of 2048 rows.
//   Each tile computes its keep flags (given, or the fused Stage-II test
//   keep1 && s2 >= tau2), a block-wide scan, and its global offset by a
//   decoupled look-back over its predecessors' published aggregates, one warp
//   reading a window of 32 predecessors at a time. Tile ids come from an
//   atomic ticket, so every predecessor has already started and publishes
//   without waiting: the look-back always ends. Its spin is bounded all the
//   same and reports OCCAM_ERR_TIMEOUT instead of hanging. The sample
//   offsets are staged in shared memory for the per-row sample lookups.
// gather_kernel: persistent grid; one warp copies one kept row of one tensor
//   with 16-byte loads / stores (exact bit copy).
#include <cuda.h>

#include <mutex>

#include "common.cuh"
#include "kernels.cuh"
#include "nvtx.cuh"
#include "validate.cuh"

namespace occam {

namespace {
constexpr unsigned long long kFlagAgg = 1ull << 62;
constexpr unsigned long long kFlagPre = 2ull << 62;
constexpr unsigned long long kValMask = (1ull << 62) - 1;

}  // namespace

constexpr int kScanSmemSamples = 2048;  // samples whose offsets fit the scan's shared copy

// Writes the byte flags of rows r0 .. r0 + 7 (byte i of w for row r0 + i) to
// o (nullable): one 8-byte store where the rows are whole and aligned.
__device__ __forceinline__ void store_flags8(uint8_t* o, int64_t r0, int64_t R, bool whole, uint64_t w) {
  if (o == nullptr) return;
  if (whole && (reinterpret_cast<uintptr_t>(o) & 7) == 0) {
    *reinterpret_cast<uint64_t*>(o + r0) = w;
  } else {
    for (int i = 0; i < 8 && r0 + i < R; ++i) o[r0 + i] = (uint8_t)(w >> (8 * i));
  }
}

__global__ void __launch_bounds__(256) scan_kernel(ScanParams p) {
  constexpr int PER = kScanTile / 256;  // 8 rows per thread
  __shared__ int tmp[40];
  __shared__ long long s_prefix;
  __shared__ int s_tile;
  __shared__ int64_t s_ro[kScanSmemSamples + 1];
  __shared__ float s_tau[kScanSmemSamples];
  const int tid = threadIdx.x;
  if (tid == 0) s_tile = atomicAdd(p.ticket, 1);
  // the row offsets (an input) while the ticket is drawn; then, once the
  // kernel before this one has finished (its s2, thresholds and flags), the
  // samples' thresholds (Stage-II threshold mode)
  const bool ro_smem = p.bt.B <= kScanSmemSamples;
  if (ro_smem)
    for (int b = tid; b <= p.bt.B; b += blockDim.x) s_ro[b] = p.bt.row_off[b];
  pdl_wait();
  if (ro_smem && p.mode != 0)
    for (int b = tid; b < p.bt.B; b += blockDim.x) s_tau[b] = p.tau2[b];
  const int64_t* row_off = ro_smem ? s_ro : p.bt.row_off;
  const float* tau2 = ro_smem ? s_tau : p.tau2;
  __syncthreads();
  const int64_t tile = s_tile;
  const int64_t R = p.bt.total_rows;
  const int64_t r_first = tile * kScanTile + (int64_t)tid * PER;
  // flags of my rows. Their inputs are loaded first, all together (one
  // memory round trip: 8-byte loads of the byte flags and 16-byte loads of
  // s2 where the rows are whole and aligned), then tested.
  uint64_t in_a = 0, in_b = 0;  // byte i: row r_first + i (mode 0: keep_in, role; mode 1: role, keep1)
  float in_s[PER];              // mode 1: s2
  const uint8_t* pa = p.mode == 0 ? p.keep_in : p.role;
  const uint8_t* pb = p.mode == 0 ? p.role : p.keep1;
  const bool whole = r_first + PER <= R;
  const bool vec = whole && ((reinterpret_cast<uintptr_t>(pa) | reinterpret_cast<uintptr_t>(pb)) & 7) == 0 &&
                   (p.mode == 0 || (reinterpret_cast<uintptr_t>(p.s2) & 15) == 0);
  if (vec) {
    in_a = *reinterpret_cast<const uint64_t*>(pa + r_first);
    if (pb) in_b = *reinterpret_cast<const uint64_t*>(pb + r_first);
    if (p.mode != 0) {
      const float4 s0 = *reinterpret_cast<const float4*>(p.s2 + r_first);
      const float4 s1 = *reinterpret_cast<const float4*>(p.s2 + r_first + 4);
      in_s[0] = s0.x; in_s[1] = s0.y; in_s[2] = s0.z; in_s[3] = s0.w;
      in_s[4] = s1.x; in_s[5] = s1.y; in_s[6] = s1.z; in_s[7] = s1.w;
    }
  } else {
#pragma unroll
    for (int i = 0; i < PER; ++i) {
      const int64_t r = r_first + i;
      const bool ok = r < R;
      in_a |= (uint64_t)(ok ? pa[r] : 0) << (8 * i);
      in_b |= (uint64_t)(ok && pb ? pb[r] : 0) << (8 * i);
      in_s[i] = ok && p.mode != 0 ? p.s2[r] : 0.f;
    }
  }
  unsigned kmask = 0, vmask = 0;
  int samp = -1;
  int64_t samp_end = 0;
  if (r_first < R) {
    samp = upper_interval(row_off, p.bt.B, r_first);
    if (!in_bounds(samp >= 0 && samp < p.bt.B, p.status, kSiteScanSample)) samp = 0;
    samp_end = row_off[samp + 1];
  }
  uint64_t kw = 0, nw = 0;  // keep2 and near bytes of my rows
#pragma unroll
  for (int i = 0; i < PER; ++i) {
    const int64_t r = r_first + i;
    bool k = false, vis = false, nr = false;
    if (r < R) {
      while (r >= samp_end) { ++samp; samp_end = row_off[samp + 1]; }
      if (p.mode == 0) {
        k = (in_a >> (8 * i) & 0xffu) != 0;
        vis = k && (p.role == nullptr || (in_b >> (8 * i) & 0xffu) == 0);
      } else if ((in_a >> (8 * i) & 0xffu) != 0) {  // a register row
        k = p.keep_registers != 0;
      } else {
        const float sv = in_s[i], t = tau2[samp];
        const bool s1row = (in_b >> (8 * i) & 0xffu) != 0;
        k = s1row && (sv >= t);
        vis = k;
        // near-threshold flag of a visual S1 row: the same fp32 tau as the test
        nr = s1row && fabsf(sv - t) <= p.near_rel * fabsf(t);
      }
    }
    kw |= (uint64_t)k << (8 * i);
    nw |= (uint64_t)nr << (8 * i);
    kmask |= (unsigned)k << i;
    vmask |= (unsigned)vis << i;
  }
  if (p.mode != 0) {
    // keep2 and the near flags of my rows, 8 bytes at a time where aligned
    store_flags8(p.keep_out, r_first, R, whole, kw);
    store_flags8(p.near_out, r_first, R, whole, nw);
  }
  const int cnt = __popc(kmask);
  int tile_total;
  const int pos = block_exclusive_scan(cnt, tmp, &tile_total);

  if (tid < 32) {
    // warp-wide look-back: lane l reads predecessor (hi - l); the window
    // moves back by 32 until it holds an inclusive prefix (tile "-1" counts
    // as an inclusive prefix of 0)
    const int lane = tid;
    long long excl = 0;
    if (tile == 0) {
      if (lane == 0) st_release_u64(&p.tile_state[0], kFlagPre | (unsigned long long)tile_total);
    } else {
      if (lane == 0) st_release_u64(&p.tile_state[tile], kFlagAgg | (unsigned long long)tile_total);
      int64_t hi = tile - 1;
      bool timed_out = false;
      uint32_t spins = 0;
      while (true) {
        const int64_t q = hi - lane;
        const unsigned long long v = q >= 0 ? ld_acquire_u64(&p.tile_state[q]) : kFlagPre;
        if (!__all_sync(0xffffffffu, (v & (kFlagAgg | kFlagPre)) != 0)) {
          if (++spins > kSpinLimit) {
            timed_out = true;
            break;
          }
          __nanosleep(32);
          continue;
        }
        const unsigned pre = __ballot_sync(0xffffffffu, (v & kFlagPre) != 0);
        const int first = pre ? __ffs(pre) - 1 : 32;  // nearest predecessor with an inclusive prefix
        long long val = lane <= first ? (long long)(v & kValMask) : 0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) val += __shfl_xor_sync(0xffffffffu, val, o);
        excl += val;
        if (pre) break;
        hi -= 32;
      }
      if (lane == 0) {
        if (timed_out) set_status(p.status, OCCAM_ERR_TIMEOUT);
        st_release_u64(&p.tile_state[tile], kFlagPre | (unsigned long long)(excl + tile_total));
      }
    }
    if (lane == 0) s_prefix = excl;
  }
  __syncthreads();
  const int64_t base = s_prefix + pos;
  // out_index + capacity
  {
    int64_t o = base;
    bool overflow = false;
    for (int i = 0; i < PER; ++i) {
      if (kmask >> i & 1) {
        if (o < p.capacity) p.out_index[o] = (int32_t)(r_first + i);
        else overflow = true;
        ++o;
      }
    }
    if (overflow) set_status(p.status, OCCAM_ERR_CAPACITY);
  }
  // per-sample counts: a thread's rows may span several samples
  {
    int s = (r_first < R) ? upper_interval(row_off, p.bt.B, r_first) : -1;
    if (s >= 0 && !in_bounds(s < p.bt.B, p.status, kSiteScanSample)) s = 0;
    int64_t send = (s >= 0) ? row_off[s + 1] : 0;
    int ck = 0, cv = 0;
    for (int i = 0; i < PER; ++i) {
      const int64_t r = r_first + i;
      if (r >= R) break;
      while (r >= send) {
        if (ck) atomicAdd(&p.count_out[s], ck);
        if (cv && p.count_vis) atomicAdd(&p.count_vis[s], cv);
        ck = cv = 0;
        ++s;
        send = row_off[s + 1];
      }
      ck += (kmask >> i) & 1;
      cv += (vmask >> i) & 1;
    }
    if (s >= 0) {
      if (ck) atomicAdd(&p.count_out[s], ck);
      if (cv && p.count_vis) atomicAdd(&p.count_vis[s], cv);
    }
  }
  // out_off[b] for every sample whose first row lies in my rows
  if (r_first < R) {
    const int64_t r_end = min(r_first + PER, R);
    // empty samples share their start row with the next one: visit every b
    // whose first row lies in [r_first, r_end)
    int bb = lower_bound_off(row_off, p.bt.B, r_first);
    for (; bb < p.bt.B && row_off[bb] < r_end; ++bb) {
      const int before = __popc(kmask & ((1u << (int)(row_off[bb] - r_first)) - 1u));
      p.out_off[bb] = base + before;
    }
  }
  // the last tile also writes out_off for the samples that start at the end
  const int64_t ntiles = (R + kScanTile - 1) / kScanTile;
  if (tile == ntiles - 1 && tid == 0) {
    const long long total = s_prefix + tile_total;
    for (int bb = p.bt.B; bb >= 0 && row_off[bb] >= R; --bb) p.out_off[bb] = total;
  }
  pdl_trigger();  // the gather kernel may be scheduled (it waits for these results)
}

// A batch with no rows at all has no scan tile: its offsets are all zero.
__global__ void offsets_fix_kernel(ScanParams p) {
  for (int b = threadIdx.x; b <= p.bt.B; b += blockDim.x) p.out_off[b] = 0;
}

__global__ void __launch_bounds__(256) gather_kernel(GatherParams p) {
  constexpr int U = 8;
  const int lane = threadIdx.x & 31;
  const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  pdl_wait();  // the scan's offsets and row list
  const int64_t total = min(p.out_off[p.B], p.capacity);
  const int64_t items = total * p.n_tensors;
  for (int64_t w = gw; w < items; w += nw) {
    const int64_t k = w / p.n_tensors;
    const int t = (int)(w - k * p.n_tensors);
    const int64_t rbytes = p.row_bytes[t];
    const int64_t row = p.out_index[k];
    if (!in_bounds(row >= 0 && row < p.src_rows, p.status, kSiteGatherRow)) continue;
    const unsigned char* src = p.src[t] + row * rbytes;
    unsigned char* dst = p.dst[t] + k * rbytes;
    int64_t off = (int64_t)lane * 16;
    for (; off + (U - 1) * 512 < rbytes; off += U * 512) {
      uint4 v[U];
#pragma unroll
      for (int u = 0; u < U; ++u) v[u] = ldg_stream(src + off + u * 512);
#pragma unroll
      for (int u = 0; u < U; ++u) stg_stream(dst + off + u * 512, v[u]);
    }
    for (; off < rbytes; off += 512) stg_stream(dst + off, ldg_stream(src + off));
  }
}

// stage_rows_kernel: persistent grid; one warp per row position p of the
// batch, copying row dense[p] (8 KB for H2 = 32) when p lies in its sample's
// S1 list. With a host source the loads cross the host link, so each lane
// keeps U 16-byte loads in flight.
__global__ void __launch_bounds__(256) stage_rows_kernel(StageRowsParams p) {
  constexpr int U = 8;
  const int lane = threadIdx.x & 31;
  const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int64_t rbytes = p.row_bytes;
  for (int64_t pos = gw; pos < p.bt.total_rows; pos += nw) {
    const int b = upper_interval(p.bt.row_off, p.bt.B, pos);
    if (pos - p.bt.row_off[b] >= p.n1[b]) continue;
    const int64_t row = p.dense[pos];
    if (!in_bounds(row >= 0 && row < p.bt.total_rows, p.status, kSiteStageRow)) continue;
    const unsigned char* src = p.src + row * rbytes;
    unsigned char* dst = p.dst + row * rbytes;
    int64_t off = (int64_t)lane * 16;
    for (; off + (U - 1) * 512 < rbytes; off += U * 512) {
      uint4 v[U];
#pragma unroll
      for (int u = 0; u < U; ++u) v[u] = ldg_stream(src + off + u * 512);
#pragma unroll
      for (int u = 0; u < U; ++u) *reinterpret_cast<uint4*>(dst + off + u * 512) = v[u];
    }
    for (; off < rbytes; off += 512) *reinterpret_cast<uint4*>(dst + off) = ldg_stream(src + off);
  }
}

// registers_kernel: one CTA per segment. For each register channel in turn,
// the CTA takes the max over the segment's visual rows (a thread-strided
// pass, then a block max), writes it into the channel of every register row
// and zeroes the channel on the visual rows. Values are compared as floats;
// the written max is one of the bf16 inputs, so results are exact.
__global__ void __launch_bounds__(256) registers_kernel(RegistersParams p) {
  __shared__ float wmax[8];
  const int seg = blockIdx.x;
  const int tid = threadIdx.x;
  const int64_t r0 = p.bt.seg_off[seg], r1 = p.bt.seg_off[seg + 1];
  const int32_t g0 = p.bt.reg_off[seg], g1 = p.bt.reg_off[seg + 1];
  for (int j = 0; j < p.n_k; ++j) {
    const int64_t k = p.k_reg[j];
    float m = -INFINITY;
    for (int64_t r = r0 + tid; r < r1; r += blockDim.x)
      if (p.role[r] == 0) m = fmaxf(m, __bfloat162float(p.h[r * p.channels + k]));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    if ((tid & 31) == 0) wmax[tid >> 5] = m;
    __syncthreads();
    float mx = wmax[0];
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) mx = fmaxf(mx, wmax[w]);
    // a segment without visual rows leaves its registers as they are
    if (mx != -INFINITY)
      for (int i = g0 + tid; i < g1; i += blockDim.x) p.h[(int64_t)p.bt.reg_idx[i] * p.channels + k] = __float2bfloat16_rn(mx);
    for (int64_t r = r0 + tid; r < r1; r += blockDim.x)
      if (p.role[r] == 0) p.h[r * p.channels + k] = __float2bfloat16_rn(0.f);
    __syncthreads();
  }
}

// Rows the Stage-II test keeps at lam, as the library applies it: candidates
// (key bit 31) with s2 >= fl(lam * ref2) in fp32. Block-wide; every thread
// of the CTA calls it and gets the total.
__device__ int lambda2_kept(const Lambda2Params& p, float lam, int* s_cnt) {
  if (threadIdx.x == 0) *s_cnt = 0;
  __syncthreads();
  int c = 0;
  for (int64_t r = threadIdx.x; r < p.bt.total_rows; r += blockDim.x) {
    if (p.keys[r] >> 31) {
      const int b = upper_interval(p.bt.row_off, p.bt.B, r);
      c += p.s2[r] >= __fmul_rn(lam, p.ref2[b]) ? 1 : 0;
    }
  }
  c = __reduce_add_sync(0xffffffffu, c);
  if ((threadIdx.x & 31) == 0) atomicAdd(s_cnt, c);
  __syncthreads();
  const int tot = *s_cnt;
  __syncthreads();
  return tot;
}

// lambda2 budget matching (App. A, Eq. 19), over all SMs. Each candidate
// row (a visual S1 row of a sample with ref2 > 0) gets the key 2^31 |
// bits(s2 / ref2), with an IEEE round-to-nearest fp32 quotient >= 0 whose bit
// pattern orders like its value; every other row gets key 0, below every
// candidate. The K-th largest key is found eleven bits at a time (bits
// 31-21, 20-10, 9-0): a grid-wide histogram of the keys that match the digits
// chosen so far, then one CTA picks the bucket where the running count from
// the top reaches K. With K <= the candidate count the result is the K-th
// largest candidate ratio. The rule applies lambda2 as one fp32 product
// (s2 >= fl(lambda2 * ref2)), whose rounding can disagree with the
// quotient's by an ulp or two: the kept counts of the ratio and its
// neighbours up to kL2Window fp32 steps either way are taken in one more
// grid pass, and the largest of them that keeps at least K rows is the
// result (single steps beyond the window, should the answer lie there).
namespace {
struct L2Sel {
  uint32_t prefix;  // the key's digits chosen so far
  int32_t k;        // rank still sought among the keys matching prefix
  int32_t done;     // the result is already written (K <= 0 or K > candidates)
  int32_t n;        // candidates
  unsigned long long kept[2 * kL2Window + 1];  // kept counts of lambda0 stepped by -W..W
  uint32_t hist[3][kL2Digits];
};
static_assert(sizeof(L2Sel) <= kL2SelBytes, "lambda2 selection scratch");

__device__ __forceinline__ L2Sel* l2sel(const Lambda2Params& p) { return reinterpret_cast<L2Sel*>(p.sel); }

// the level's digit shift and the mask of the digits above it
__device__ __forceinline__ int l2_shift(int level) { return level == 0 ? 21 : level == 1 ? 10 : 0; }
__device__ __forceinline__ uint32_t l2_mask_above(int level) {
  return level == 0 ? 0u : level == 1 ? 0xFFE00000u : 0xFFFFFC00u;
}

// lambda0 stepped by j fp32 steps (j < 0: down, toward 0)
__device__ __forceinline__ float l2_step(float lam, int j) {
  for (; j < 0; ++j) lam = nextafterf(lam, 0.f);
  for (; j > 0; --j) lam = nextafterf(lam, __int_as_float(0x7f800000));
  return lam;
}
}  // namespace

// keys of every row and the histogram of their top digit
__global__ void __launch_bounds__(256) l2_keys_kernel(Lambda2Params p) {
  __shared__ uint32_t h[kL2Digits];
  L2Sel* st = l2sel(p);
  for (int i = threadIdx.x; i < kL2Digits; i += blockDim.x) h[i] = 0;
  __syncthreads();
  const int64_t R = p.bt.total_rows;
  int cnt = 0;
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < R; r += (int64_t)gridDim.x * blockDim.x) {
    const int b = upper_interval(p.bt.row_off, p.bt.B, r);
    const float ref = p.ref2[b];
    uint32_t key = 0;
    if (p.keep1[r] && p.role[r] == 0 && ref > 0.f) {
      key = 0x80000000u | __float_as_uint(__fdiv_rn(p.s2[r], ref));
      atomicAdd(&h[key >> 21], 1u);
      ++cnt;
    }
    p.keys[r] = key;
  }
  cnt = __reduce_add_sync(0xffffffffu, cnt);
  if ((threadIdx.x & 31) == 0 && cnt) atomicAdd(&st->n, cnt);
  __syncthreads();
  for (int i = threadIdx.x; i < kL2Digits; i += blockDim.x)
    if (h[i]) atomicAdd(&st->hist[0][i], h[i]);
}

// histogram of the level's digit over the keys that match the digits above it
__global__ void __launch_bounds__(256) l2_hist_kernel(Lambda2Params p, int level) {
  __shared__ uint32_t h[kL2Digits];
  L2Sel* st = l2sel(p);
  if (st->done) return;
  for (int i = threadIdx.x; i < kL2Digits; i += blockDim.x) h[i] = 0;
  __syncthreads();
  const uint32_t prefix = st->prefix, mask = l2_mask_above(level);
  const int shift = l2_shift(level);
  const int64_t R = p.bt.total_rows;
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < R; r += (int64_t)gridDim.x * blockDim.x) {
    const uint32_t key = p.keys[r];
    if ((key & mask) == prefix && (key >> 31)) atomicAdd(&h[(key >> shift) & (kL2Digits - 1)], 1u);
  }
  __syncthreads();
  for (int i = threadIdx.x; i < kL2Digits; i += blockDim.x)
    if (h[i]) atomicAdd(&st->hist[level][i], h[i]);
}

// one CTA of 1,024 threads: the bucket of the level's histogram where the
// count from the top reaches k (thread t holds buckets 2047 - 2t and 2046 - 2t)
__global__ void __launch_bounds__(1024) l2_select_kernel(Lambda2Params p, int level) {
  __shared__ int tmp[40];
  L2Sel* st = l2sel(p);
  const int tid = threadIdx.x;
  if (level == 0) {
    const int n = st->n;
    if (tid == 0 && p.n_candidates) *p.n_candidates = n;
    if (p.target <= 0 || p.target > n) {
      // K <= 0: no lambda2 keeps nothing but +inf; K > n: 0 keeps every candidate
      if (tid == 0) {
        *p.lambda2 = p.target <= 0 ? __int_as_float(0x7f800000) : 0.f;
        st->done = 1;
      }
      return;
    }
  }
  if (st->done) return;
  const int k = level == 0 ? (int)p.target : st->k;
  const uint32_t* hist = st->hist[level];
  const int hi = kL2Digits - 1 - 2 * tid, lo = hi - 1;
  const int chi = (int)hist[hi], clo = (int)hist[lo];
  int total;
  const int above = block_exclusive_scan(chi + clo, tmp, &total);
  if (above < k && k <= above + chi + clo) {
    const int bucket = above + chi >= k ? hi : lo;
    const int k_rest = bucket == hi ? k - above : k - above - chi;
    const uint32_t prefix = (level == 0 ? 0u : st->prefix) | ((uint32_t)bucket << l2_shift(level));
    st->prefix = prefix;
    st->k = k_rest;
  }
}

// kept counts of the selected ratio and its neighbours, one grid pass
__global__ void __launch_bounds__(256) l2_window_kernel(Lambda2Params p) {
  L2Sel* st = l2sel(p);
  if (st->done) return;
  constexpr int NW = 2 * kL2Window + 1;
  const float lam0 = __uint_as_float(st->prefix & 0x7fffffffu);
  float lam[NW];
#pragma unroll
  for (int j = 0; j < NW; ++j) lam[j] = l2_step(lam0, j - kL2Window);
  int c[NW];
#pragma unroll
  for (int j = 0; j < NW; ++j) c[j] = 0;
  const int64_t R = p.bt.total_rows;
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < R; r += (int64_t)gridDim.x * blockDim.x) {
    if (p.keys[r] >> 31) {
      const int b = upper_interval(p.bt.row_off, p.bt.B, r);
      const float s = p.s2[r], ref = p.ref2[b];
#pragma unroll
      for (int j = 0; j < NW; ++j) c[j] += s >= __fmul_rn(lam[j], ref) ? 1 : 0;
    }
  }
#pragma unroll
  for (int j = 0; j < NW; ++j) {
    const int v = __reduce_add_sync(0xffffffffu, c[j]);
    if ((threadIdx.x & 31) == 0 && v) atomicAdd(&st->kept[j], (unsigned long long)v);
  }
}

// one CTA of 1,024 threads: the largest lambda2 of the window whose product
// test keeps at least K rows; beyond the window, single fp32 steps as before
__global__ void __launch_bounds__(1024) l2_finish_kernel(Lambda2Params p) {
  __shared__ int s_kept;
  __shared__ float s_lam;
  L2Sel* st = l2sel(p);
  if (st->done) return;
  constexpr int NW = 2 * kL2Window + 1;
  const int64_t K = p.target;
  const float lam0 = __uint_as_float(st->prefix & 0x7fffffffu);
  if ((int64_t)st->kept[0] < K) {
    // below the window: down while fewer than K are kept (kept(0) counts every candidate)
    if (threadIdx.x == 0) s_lam = l2_step(lam0, -kL2Window);
    __syncthreads();
    for (int it = 0; it < 64; ++it) {
      const float lam = nextafterf(s_lam, 0.f);
      if (lambda2_kept(p, lam, &s_kept) >= K) {
        if (threadIdx.x == 0) s_lam = lam;
        break;
      }
      if (threadIdx.x == 0) s_lam = lam;
      __syncthreads();
    }
  } else if ((int64_t)st->kept[NW - 1] >= K) {
    // above the window: up while the next value still keeps K
    if (threadIdx.x == 0) s_lam = l2_step(lam0, kL2Window);
    __syncthreads();
    for (int it = 0; it < 64; ++it) {
      const float up = nextafterf(s_lam, __int_as_float(0x7f800000));
      if (lambda2_kept(p, up, &s_kept) < K) break;
      if (threadIdx.x == 0) s_lam = up;
      __syncthreads();
    }
  } else {
    if (threadIdx.x == 0) {
      int j = NW - 1;
      while ((int64_t)st->kept[j] < K) --j;  // kept is non-increasing in lambda2; kept[0] >= K
      s_lam = l2_step(lam0, j - kL2Window);
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) *p.lambda2 = s_lam;
}

}  // namespace occam

// ============================================================================
// occam_compact_noalloc: occam_compact for callers that cannot allocate
// device memory. Its scratch (the scan's tile states, the tile ticket and a
// status word) lives in the file-scope array below instead of a caller
// workspace. Every GPU that loads this library holds the array (64.25 KiB)
// until the process exits; all calls on a device share it.
// ============================================================================
namespace {

constexpr int64_t kNoAllocMaxTiles = 8192;  // total_rows <= 8192 * 2048 = 16,777,216
constexpr int kNoAllocMaxDevices = 64;

// [0, kNoAllocMaxTiles): tile states; then one int32 ticket and one int32 status
static __device__ __align__(256) unsigned long long g_noalloc_scratch[kNoAllocMaxTiles + 32];

// The array's device address belongs to the CUDA context that loaded this
// module: it is looked up once per context (with its device current) and
// cached under the context's unique id, so a context created later on the
// same device (after cudaDeviceReset, or a driver-API context) gets its own
// lookup instead of a stale address.
struct NoAllocEntry {
  unsigned long long ctx_id = 0;
  void* ptr = nullptr;
  int sms = 0;
};
std::mutex g_noalloc_mu;
NoAllocEntry g_noalloc[kNoAllocMaxDevices];
int g_noalloc_next = 0;

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

// The unique id of the current context (0 if there is none or the driver
// cannot say).
unsigned long long current_ctx_id() {
  static CtxGetCurrentFn get_cur = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_cur = reinterpret_cast<CtxGetCurrentFn>(f);
    f = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(f);
  });
  CUcontext c = nullptr;
  unsigned long long id = 0;
  if (!get_cur || !get_id || get_cur(&c) != CUDA_SUCCESS || c == nullptr || get_id(c, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// Device address of the static scratch in the current context, and the
// device's SM count.
int noalloc_scratch(void** ptr, int* sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return OCCAM_ERR_CUDA;
  // the runtime creates the device's context on its first use: look the
  // address up first, then read the id of the context it belongs to
  void* p = nullptr;
  std::lock_guard<std::mutex> lock(g_noalloc_mu);
  unsigned long long id = current_ctx_id();
  if (id != 0) {
    for (const NoAllocEntry& e : g_noalloc) {
      if (e.ctx_id == id) {
        *ptr = e.ptr;
        *sms = e.sms;
        return OCCAM_OK;
      }
    }
  }
  if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || p == nullptr) return OCCAM_ERR_CUDA;
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
  if (id == 0) id = current_ctx_id();
  if (id != 0) {
    // a new context: one cache slot (round robin once all are taken)
    NoAllocEntry& e = g_noalloc[g_noalloc_next];
    g_noalloc_next = (g_noalloc_next + 1) % kNoAllocMaxDevices;
    e.ctx_id = id;
    e.ptr = p;
    e.sms = n;
  }
  *ptr = p;
  *sms = n;
  return OCCAM_OK;
}

}  // namespace

extern "C" int occam_compact_noalloc(const occam_batch* b, const uint8_t* keep, int32_t n_tensors,
                                     const void* const* src, const int64_t* row_bytes, void* const* dst,
                                     int64_t capacity_rows, int32_t* out_index, int32_t* count_out,
                                     int64_t* out_off, occam_stream_t stream) {
  const NvtxRange nvtx("occam_compact_noalloc");
  occam::launch_counter() = 0;
  using namespace occam;
  // the same checks as occam_compact's, then the limit of the fixed scratch
  const int rc_batch = check_batch(b);
  if (rc_batch != OCCAM_OK) return rc_batch;
  const int rc_gather = check_gather(n_tensors, src, row_bytes, dst);
  if (rc_gather != OCCAM_OK) return rc_gather;
  if (!keep || !count_out || !out_off || capacity_rows < 0 || (capacity_rows > 0 && !out_index))
    return OCCAM_ERR_INVALID_ARG;
  const int64_t ntiles = (b->total_rows + kScanTile - 1) / kScanTile;
  if (ntiles > kNoAllocMaxTiles) return OCCAM_ERR_UNSUPPORTED;  // more rows than the static scratch covers
  void* scratch = nullptr;
  int sms = 0;
  const int rc = noalloc_scratch(&scratch, &sms);
  if (rc != OCCAM_OK) return rc;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  unsigned long long* tiles = static_cast<unsigned long long*>(scratch);
  int32_t* ticket = reinterpret_cast<int32_t*>(tiles + kNoAllocMaxTiles);
  int* status = reinterpret_cast<int*>(ticket + 1);
  // the array keeps the previous call's contents: clear what must start at zero
  if (cudaMemsetAsync(tiles, 0, ntiles * 8, st) != cudaSuccess) return OCCAM_ERR_CUDA;
  if (cudaMemsetAsync(ticket, 0, 8, st) != cudaSuccess) return OCCAM_ERR_CUDA;
  if (cudaMemsetAsync(count_out, 0, b->B * 4, st) != cudaSuccess) return OCCAM_ERR_CUDA;
  ScanParams p;
  p.bt.B = b->B;
  p.bt.S_tot = b->S_tot;
  p.bt.total_rows = b->total_rows;
  p.bt.total_text = b->total_text;
  p.bt.row_off = b->row_off;
  p.bt.seg_off = b->seg_off;
  p.bt.seg_first = b->seg_first;
  p.bt.seg_sample = b->seg_sample;
  p.bt.reg_idx = b->reg_idx;
  p.bt.reg_off = b->reg_off;
  p.bt.text_off = b->text_off;
  p.mode = 0;
  p.keep_in = keep;
  p.role = nullptr;
  p.keep1 = nullptr;
  p.s2 = nullptr;
  p.tau2 = nullptr;
  p.keep_registers = 0;
  p.keep_out = nullptr;
  p.capacity = capacity_rows;
  p.out_index = out_index;
  p.count_out = count_out;
  p.count_vis = nullptr;
  p.out_off = out_off;
  p.tile_state = tiles;
  p.ticket = ticket;
  p.ntiles = ntiles;
  p.status = status;
  scan_kernel<<<(unsigned)ntiles, 256, 0, st>>>(p);
  count_launch();
  if (n_tensors > 0) {
    GatherParams g;
    g.n_tensors = n_tensors;
    for (int t = 0; t < OCCAM_MAX_GATHER; ++t) {
      g.src[t] = t < n_tensors ? static_cast<const unsigned char*>(src[t]) : nullptr;
      g.dst[t] = t < n_tensors ? static_cast<unsigned char*>(dst[t]) : nullptr;
      g.row_bytes[t] = t < n_tensors ? row_bytes[t] : 0;
    }
    g.out_index = out_index;
    g.out_off = out_off;
    g.B = b->B;
    g.capacity = capacity_rows;
    g.src_rows = b->total_rows;
    g.status = status;
    gather_kernel<<<sms * 4, 256, 0, st>>>(g);
    count_launch();
  }
  return cudaGetLastError() == cudaSuccess ? OCCAM_OK : OCCAM_ERR_CUDA;
}
