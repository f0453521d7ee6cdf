// common.cuh -- shared device helpers and internal parameter blocks for the
// OccamToken prune kernels (sm_103a). Nothing here is part of the C ABI.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/occam.h"

namespace occam {

// Kernels launched by the current host thread since the entry point it is in
// began (each entry point resets it; occam_last_call_kernels reports it).
int& launch_counter();
inline void count_launch(int n = 1) { launch_counter() += n; }

constexpr int kWarp = 32;

// ---------------------------------------------------------------- status word
// The first device-side error wins; later ones are dropped.
__device__ __forceinline__ void set_status(int* status, int code) {
  if (status) atomicCAS(status, 0, code);
}

}  // namespace occam

#include "check.cuh"

namespace occam {

// ---------------------------------------------------------------- bf16 helpers
__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xffff0000u); }

// 16-byte read-only global load that is not kept in L1 (streamed once).
__device__ __forceinline__ uint4 ldg_stream(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ void stg_stream(void* p, uint4 v) {
  asm volatile("st.global.L1::no_allocate.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y),
               "r"(v.z), "r"(v.w)
               : "memory");
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ int warp_sum_i(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Block-wide exclusive scan of one int per thread (blockDim.x a multiple of 32,
// at most 1024). `tmp` holds >= 33 ints of shared memory. Returns the
// exclusive prefix; *total receives the block sum. Contains __syncthreads.
__device__ __forceinline__ int block_exclusive_scan(int v, int* tmp, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int n = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += n;
  }
  if (lane == 31) tmp[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    int w = lane < nw ? tmp[lane] : 0;
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      int n = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += n;
    }
    if (lane < nw) tmp[lane] = wi - w;
    if (lane == nw - 1) tmp[32] = wi;
  }
  __syncthreads();
  int res = tmp[warp] + incl - v;
  *total = tmp[32];
  __syncthreads();
  return res;
}

// 2^x with the hardware approximation (relative error about 2^-22),
// flushing subnormal results to zero; 2^-inf = 0
__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Programmatic dependent launch. A kernel launched with the programmatic
// stream-serialization attribute may start once every CTA of the kernel
// before it in the stream has called pdl_trigger() (or exited); until it
// calls pdl_wait() it may read only what was complete before that kernel
// started (inputs, earlier kernels' results). pdl_wait() returns once the
// previous kernel has finished and its writes are visible. Both are no-ops
// for kernels launched without the attribute.
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// N exclusive prefix sums over the block at once (three barriers in all, as
// for one): excl[k] = sum of v[k] over the threads before this one, total[k]
// = the block's sum. tmp: N * 33 ints of shared memory.
template <int N>
__device__ __forceinline__ void block_exclusive_scan_n(const int (&v)[N], int (&excl)[N], int (&total)[N], int* tmp) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int incl[N];
#pragma unroll
  for (int k = 0; k < N; ++k) {
    incl[k] = v[k];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int n = __shfl_up_sync(0xffffffffu, incl[k], o);
      if (lane >= o) incl[k] += n;
    }
    if (lane == 31) tmp[k * 33 + warp] = incl[k];
  }
  __syncthreads();
  if (warp == 0) {
#pragma unroll
    for (int k = 0; k < N; ++k) {
      const int w = lane < nw ? tmp[k * 33 + lane] : 0;
      int wi = w;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int n = __shfl_up_sync(0xffffffffu, wi, o);
        if (lane >= o) wi += n;
      }
      if (lane < nw) tmp[k * 33 + lane] = wi - w;
      if (lane == nw - 1) tmp[k * 33 + 32] = wi;
    }
  }
  __syncthreads();
#pragma unroll
  for (int k = 0; k < N; ++k) {
    excl[k] = tmp[k * 33 + warp] + incl[k] - v[k];
    total[k] = tmp[k * 33 + 32];
  }
  __syncthreads();
}

// Index of the interval of `off` ([n+1] ascending) that holds x: off[i] <= x < off[i+1].
template <typename T>
__device__ __forceinline__ int upper_interval(const T* off, int n, int64_t x) {
  int lo = 0, hi = n;  // invariant: off[lo] <= x < off[hi]
  while (hi - lo > 1) {
    int mid = (lo + hi) >> 1;
    if ((int64_t)off[mid] <= x) lo = mid; else hi = mid;
  }
  return lo;
}

// First index i in [0, n] with off[i] >= x (off ascending, [n+1] entries).
template <typename T>
__device__ __forceinline__ int lower_bound_off(const T* off, int n, int64_t x) {
  int lo = 0, hi = n + 1;
  while (lo < hi) {
    int mid = (lo + hi) >> 1;
    if ((int64_t)off[mid] < x) lo = mid + 1; else hi = mid;
  }
  return lo;
}

// ---------------------------------------------------------------- async copies
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// mbarrier + bulk (TMA 1-D) copy global -> shared
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}
// Bounded wait on phase `parity`; returns false if it gave up.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, uint32_t max_iter) {
  uint32_t done = 0;
  for (uint32_t it = 0; it < max_iter; ++it) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    if (done) return true;
  }
  return false;
}
__device__ __forceinline__ void bulk_g2s(void* smem, const void* gmem, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(smem)),
      "l"(gmem), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

// release store / acquire load of a 64-bit flag word (GPU scope)
__device__ __forceinline__ void st_release_u64(unsigned long long* p, unsigned long long v) {
  asm volatile("st.release.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

// ---------------------------------------------------------------- internal parameter blocks
// Workspace carve-up (byte offsets from the workspace base; see ws_layout()).
struct WsLayout {
  size_t status, counters, role, keep1, s1, s2, ref1, dense, n1, n1_vis;
  size_t itemsHS, ppart, itemA_off, itemB_off, stats2, refpart, ref2, tau2, done, scan_state, seg_state, stats1, itemsF, itemsF8, itemsF16,
      slot_off;
  size_t l2sel;                 // lambda2 selection scratch (kL2SelBytes)
  size_t zero_begin, zero_end;  // the accumulators every prune call zeroes (one contiguous range)
  size_t total;
  int64_t maxA, maxB, maxF, maxSlots, scan_tiles, stats1_rows;
};

// counters block (int32 slots)
enum {
  CNT_DENSE_DONE = 0,
  CNT_SCAN_TICKET = 1,
  CNT_NA = 2,
  CNT_NB = 3,
  CNT_NF = 4,
  CNT_NF8 = 5,
  CNT_QUEUE4 = 6,  // next fused Stage-II item (4-CTA clusters)
  CNT_QUEUE8 = 7,  // next fused Stage-II item (8-CTA clusters)
  CNT_SEG_TICKET = 8,  // Stage-I finalize: segment order
  CNT_NF16 = 9,
  CNT_QUEUE16 = 10,    // next fused Stage-II item (16-CTA clusters)
  CNT_MUT = 11,        // [2] next mutual Stage-I item of each pass
  CNT_NHS = 13,        // Stage-II text tiles split over head groups (merge items)
  CNT_SLOTS = 14
};

constexpr int kTextTile = 64;    // Stage-II text rows per item of the two-pass score pass
constexpr int kStatsTile = 128;  // Stage-II text rows per item of the two-pass statistics pass
constexpr int kHeadGroup = 4;    // Stage-II heads per stats item
constexpr int kStatSplits = 16;  // at most this many key ranges per (text tile, head group) in the stats pass
constexpr int kKeyChunk = 128;   // Stage-II image keys per score item
constexpr int kScanTile = 2048;  // compaction rows per scan tile (256 threads x 8)
constexpr uint32_t kSpinLimit = 1u << 22;

struct BatchDev {
  int B, S_tot;
  int64_t total_rows, total_text;
  const int64_t* row_off;
  const int64_t* seg_off;
  const int32_t* seg_first;
  const int32_t* seg_sample;
  const int32_t* reg_idx;
  const int32_t* reg_off;
  const int64_t* text_off;
};

}  // namespace occam
