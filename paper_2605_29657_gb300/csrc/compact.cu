// compact.cu -- order-preserving stream compaction of the kept rows and the
// gather of their hidden / K / V rows (Algorithm 1: decoding continues on
// [S2; T]; App. A, Eq. 21: the KV cache shrinks with the kept count).
//
// scan_kernel: single pass over the batch's row space in tiles of 2048 rows.
//   Each tile computes its keep flags (given, or the fused Stage-II test
//   keep1 && s2 >= tau2), a block-wide scan, and its global offset by a
//   decoupled look-back over its predecessors' published aggregates. Tile ids
//   come from an atomic ticket, so every predecessor has already started and
//   publishes without waiting: the look-back always ends. Its spin is bounded
//   all the same and reports OCCAM_ERR_TIMEOUT instead of hanging.
// gather_kernel: persistent grid; one warp copies one kept row of one tensor
//   with 16-byte loads / stores (exact bit copy).
#include "common.cuh"
#include "kernels.cuh"

namespace occam {

namespace {
constexpr unsigned long long kFlagAgg = 1ull << 62;
constexpr unsigned long long kFlagPre = 2ull << 62;
constexpr unsigned long long kValMask = (1ull << 62) - 1;

__device__ __forceinline__ void st_release(unsigned long long* p, unsigned long long v) {
  asm volatile("st.release.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ unsigned long long ld_acquire(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
}  // namespace

__global__ void __launch_bounds__(256) scan_kernel(ScanParams p) {
  constexpr int PER = kScanTile / 256;  // 8 rows per thread
  __shared__ int tmp[40];
  __shared__ long long s_prefix;
  __shared__ int s_tile;
  const int tid = threadIdx.x;
  if (tid == 0) s_tile = atomicAdd(p.ticket, 1);
  __syncthreads();
  const int64_t tile = s_tile;
  const int64_t R = p.bt.total_rows;
  const int64_t r_first = tile * kScanTile + (int64_t)tid * PER;
  // flags of my rows
  unsigned kmask = 0, vmask = 0;
  int samp = -1;
  int64_t samp_end = 0;
  if (r_first < R) {
    samp = upper_interval(p.bt.row_off, p.bt.B, r_first);
    samp_end = p.bt.row_off[samp + 1];
  }
#pragma unroll
  for (int i = 0; i < PER; ++i) {
    const int64_t r = r_first + i;
    if (r >= R) break;
    while (r >= samp_end) { ++samp; samp_end = p.bt.row_off[samp + 1]; }
    bool k, vis;
    if (p.mode == 0) {
      k = p.keep_in[r] != 0;
      vis = k && (p.role == nullptr || p.role[r] == 0);
    } else {
      const bool reg = p.role[r] != 0;
      if (reg) {
        k = p.keep_registers != 0;
        vis = false;
      } else {
        k = (p.keep1[r] != 0) && (p.s2[r] >= p.tau2[samp]);
        vis = k;
      }
      if (p.keep_out) p.keep_out[r] = k ? 1 : 0;
    }
    kmask |= (unsigned)k << i;
    vmask |= (unsigned)vis << i;
  }
  const int cnt = __popc(kmask);
  int tile_total;
  const int pos = block_exclusive_scan(cnt, tmp, &tile_total);

  if (tid == 0) {
    long long excl = 0;
    if (tile == 0) {
      st_release(&p.tile_state[0], kFlagPre | (unsigned long long)tile_total);
    } else {
      st_release(&p.tile_state[tile], kFlagAgg | (unsigned long long)tile_total);
      int64_t q = tile - 1;
      bool timed_out = false;
      while (q >= 0) {
        unsigned long long v = 0;
        uint32_t spins = 0;
        while (true) {
          v = ld_acquire(&p.tile_state[q]);
          if (v & (kFlagAgg | kFlagPre)) break;
          if (++spins > kSpinLimit) { timed_out = true; break; }
          __nanosleep(64);
        }
        if (timed_out) break;
        excl += (long long)(v & kValMask);
        if (v & kFlagPre) break;
        --q;
      }
      if (timed_out) set_status(p.status, OCCAM_ERR_TIMEOUT);
      st_release(&p.tile_state[tile], kFlagPre | (unsigned long long)(excl + tile_total));
    }
    s_prefix = excl;
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
    int s = (r_first < R) ? upper_interval(p.bt.row_off, p.bt.B, r_first) : -1;
    int64_t send = (s >= 0) ? p.bt.row_off[s + 1] : 0;
    int ck = 0, cv = 0;
    for (int i = 0; i < PER; ++i) {
      const int64_t r = r_first + i;
      if (r >= R) break;
      while (r >= send) {
        if (ck) atomicAdd(&p.count_out[s], ck);
        if (cv && p.count_vis) atomicAdd(&p.count_vis[s], cv);
        ck = cv = 0;
        ++s;
        send = p.bt.row_off[s + 1];
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
    int bb = lower_bound_off(p.bt.row_off, p.bt.B, r_first);
    for (; bb < p.bt.B && p.bt.row_off[bb] < r_end; ++bb) {
      const int before = __popc(kmask & ((1u << (int)(p.bt.row_off[bb] - r_first)) - 1u));
      p.out_off[bb] = base + before;
    }
  }
  // the last tile also writes out_off for the samples that start at the end
  const int64_t ntiles = (R + kScanTile - 1) / kScanTile;
  if (tile == ntiles - 1 && tid == 0) {
    const long long total = s_prefix + tile_total;
    for (int bb = p.bt.B; bb >= 0 && p.bt.row_off[bb] >= R; --bb) p.out_off[bb] = total;
  }
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
  const int64_t total = min(p.out_off[p.B], p.capacity);
  const int64_t items = total * p.n_tensors;
  for (int64_t w = gw; w < items; w += nw) {
    const int64_t k = w / p.n_tensors;
    const int t = (int)(w - k * p.n_tensors);
    const int64_t rbytes = p.row_bytes[t];
    const int64_t row = p.out_index[k];
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

}  // namespace occam
