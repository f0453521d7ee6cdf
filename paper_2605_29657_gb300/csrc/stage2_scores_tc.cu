// stage2_scores_tc.cu -- the score pass of the two-pass Stage II (samples
// whose S1 keys exceed what a fused cluster holds), on the 5th-generation
// tensor cores (tcgen05 + TMEM + TMA).
//
// What it computes (Sec. 3.5, Eq. 7; App. A, Eqs. 15-16), given each text
// row's softmax statistics per head from the statistics pass (max m and sum
// z over all of its keys, in log2 units): for a work item (sample, 64 text
// rows, 128 S1 keys) the head-summed probabilities
//   P[key][row] = sum_h exp2(c q_{row,h} . k_{key,h} - m_{row,h}) / z_{row,h},
// then per key the max over the item's text rows (into s2, an order-free
// atomicMax on the fp32 bits of values >= 0) and, for register keys, the sum
// over rows (the item's share of s2(r), written to its partial slot; the
// sample's last slot writer reduces the slots in order into ref2 and tau2).
//
// Per head: the 128 keys are the MMA's A operand (one per TMEM lane, fetched
// from K2 through the S1 list by 16-byte cp.async copies into the 128-byte
// swizzled K-major layout), the 64 text queries its B operand (one TMA box
// per 64-dim K-block), and D = K Q^T (128 x 64 fp32) lands in one of two
// TMEM buffers. The key rows are scattered: per-copy TMA gathers (four rows
// a copy) left this pass bound by the copy rate, while 224 threads' cp.async
// keep two heads' key tiles in flight (the copy rate grows with the number
// of issuing warps).
// Roles (512 threads): warps 0, 2, 3 and 12-15 load the keys (warp 0 also
// issues the query TMA boxes), warp 1 issues the MMAs, warps 4-11 (two per
// TMEM lane quadrant, 32 text rows each) add each head into register
// accumulators. Operands have three stages, accumulators two. A loader
// signals a stage once its own copies landed and, through a proxy fence,
// are visible to the tensor cores. Every wait is bounded; on a timeout the
// CTA records OCCAM_ERR_TIMEOUT, lets its copies land, frees TMEM and
// returns.
#include "common.cuh"
#include "kernels.cuh"
#include "tc5.cuh"

namespace occam {

namespace s2t {
constexpr int KR = 128;                   // keys per item (MMA M, TMEM lanes)
constexpr int TR = kTextTile;             // text rows per item (MMA N)
constexpr int ABYTES = KR * 128;          // one 64-dim K-block of the key tile
constexpr int BBYTES = TR * 128;          // one 64-dim K-block of the query tile
constexpr int NST = 3;                    // operand stages
constexpr int NLOAD = 7 * 32;             // key loader threads (warps 0, 2, 3, 12-15)
constexpr int EPI0 = 4;                   // first softmax warp
constexpr int NEPI = 8;
constexpr int THREADS = 16 * 32;
constexpr int HMAX = 64;                  // heads the statistics table holds
constexpr uint64_t kLimitNs = 2000000000ull;
static_assert(TR == 64, "two softmax warps of 32 rows per quadrant");

struct Smem {
  uint8_t a[NST][2][ABYTES];   // key tile: [stage][K-block], 128-byte swizzled rows
  uint8_t b[NST][2][BBYTES];   // query tile
  float2 sst[TR][HMAX];        // per text row and head: (max, 1 / sum); rows past the text: (+inf, 0)
  float2 part[2][4][32];       // each softmax warp's (column max, register sum) per half, quadrant and lane
  float rsum[4];               // register sums of the quadrants
  int32_t kidx[KR];            // K2 row of each key of the item (padding: the first key)
  uint8_t kreg[KR];            // 1: the key is a register row
  uint64_t full[NST], empty[NST], dfull[2], dfree[2];
  uint32_t tmem_base;
  int abort;
  int last;
};
}  // namespace s2t

int s2_scores_tc_smem_bytes() { return (int)sizeof(s2t::Smem) + 1024; }
static_assert(sizeof(s2t::Smem) + 1024 <= 227 * 1024, "shared memory per CTA");

namespace {

// The sample whose items [off[b], off[b + 1]) hold item it (off ascending).
__device__ __forceinline__ int tc_item_sample(const int32_t* off, int B, int it) {
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (off[mid] <= it) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Waits for the TMEM load and ties its 32 result registers to the wait, so
// the compiler cannot move a use above it.
__device__ __forceinline__ void ld_wait32(uint32_t (&v)[32]) {
  tc::tmem_wait_ld();
  asm volatile(""
               : "+r"(v[0]), "+r"(v[1]), "+r"(v[2]), "+r"(v[3]), "+r"(v[4]), "+r"(v[5]), "+r"(v[6]), "+r"(v[7]),
                 "+r"(v[8]), "+r"(v[9]), "+r"(v[10]), "+r"(v[11]), "+r"(v[12]), "+r"(v[13]), "+r"(v[14]), "+r"(v[15]),
                 "+r"(v[16]), "+r"(v[17]), "+r"(v[18]), "+r"(v[19]), "+r"(v[20]), "+r"(v[21]), "+r"(v[22]), "+r"(v[23]),
                 "+r"(v[24]), "+r"(v[25]), "+r"(v[26]), "+r"(v[27]), "+r"(v[28]), "+r"(v[29]), "+r"(v[30]), "+r"(v[31]));
}

}  // namespace

__global__ void __launch_bounds__(s2t::THREADS, 1)
    s2_scores_tc_kernel(const __grid_constant__ CUtensorMap mapQ, Stage2Params p) {
  using namespace s2t;
  extern __shared__ unsigned char smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nB = p.counters[CNT_NB];
  if ((int)blockIdx.x >= nB) return;  // no item for this CTA: leave before touching TMEM
  const int H = p.H;
  const int kv_group = p.H / p.Hkv;
  const float c = p.scale * 1.4426950408889634f;
  const float invH = 1.0f / (float)H;
  volatile int* abort = &sm.abort;

  if (tid == 0) {
    for (int i = 0; i < NST; ++i) {
      tc::bar_init(&sm.full[i], NLOAD + 1);  // every loader, plus the query boxes' expect_tx
      tc::bar_init(&sm.empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      tc::bar_init(&sm.dfull[i], 1);
      tc::bar_init(&sm.dfree[i], NEPI);
    }
    sm.abort = 0;
    tc::bar_fence_init();
    tc::prefetch_map(&mapQ);
  }
  if (warp == 1) tc::tmem_alloc(&sm.tmem_base, 2 * TR);
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem = sm.tmem_base;

  uint32_t sg = 0;  // heads processed by this CTA (phase counter of every ring)
  for (int it = blockIdx.x; it < nB; it += gridDim.x) {
    // ---- item setup (all threads)
    const int b = tc_item_sample(p.itemB_off, p.bt.B, it);
    const int64_t t0 = p.bt.text_off[b];
    const int M = (int)(p.bt.text_off[b + 1] - t0);
    const int n_img = p.n1[b];
    const int nch = (n_img + kKeyChunk - 1) / kKeyChunk;
    const int i_in = it - p.itemB_off[b];
    const int j0 = (i_in / nch) * TR, k0 = (i_in % nch) * KR, slot = p.slot_off[b] + i_in;
    const int nq = min(TR, M - j0);
    const int nk = min(KR, n_img - k0);
    const int64_t rbase = p.bt.row_off[b];
    for (int i = tid; i < KR; i += THREADS) {
      int row = p.dense[rbase + k0 + (i < nk ? i : 0)];
      if (!in_bounds(row >= 0 && row < p.bt.total_rows, p.status, kSiteTwoPassKeyRow)) row = 0;
      sm.kidx[i] = row;
      sm.kreg[i] = (i < nk) ? p.role[row] : 0;
    }
    // the statistics pass's partials of every key range, merged: max, then
    // the sums rescaled to it
    // An entry's kStatSplits slots are 128 contiguous, 128-byte aligned
    // bytes: all are loaded at once (independent 16-byte loads, one L2 round
    // trip), slots past the sample's nsp ranges taken as empty.
    const int nsp = s2_stat_splits(n_img, M);
    for (int i = tid; i < TR * H; i += THREADS) {
      const int r = i / H, h = i - r * H;
      float2 st = make_float2(INFINITY, 0.f);
      if (r < nq) {
        const float4* ps = reinterpret_cast<const float4*>(p.stats + ((t0 + j0 + r) * H + h) * kStatSplits);
        float2 v[kStatSplits];
#pragma unroll
        for (int q = 0; q < kStatSplits / 2; ++q) {
          const float4 w = 2 * q < nsp ? __ldcg(ps + q) : make_float4(-INFINITY, 0.f, -INFINITY, 0.f);
          v[2 * q] = make_float2(w.x, w.y);
          v[2 * q + 1] = 2 * q + 1 < nsp ? make_float2(w.z, w.w) : make_float2(-INFINITY, 0.f);
        }
        float mx = -INFINITY;
#pragma unroll
        for (int s = 0; s < kStatSplits; ++s) mx = fmaxf(mx, v[s].x);
        float z = 0.f;
#pragma unroll
        for (int s = 0; s < kStatSplits; ++s)
          if (v[s].x != -INFINITY) z += v[s].y * exp2f(v[s].x - mx);
        st = make_float2(mx, 1.0f / z);
      }
      sm.sst[r][h] = st;
    }
    tc::fence_before();
    __syncthreads();
    tc::fence_after();
    if (*abort) break;  // uniform: read after the barrier

    if (warp == 0 || warp == 2 || warp == 3 || warp >= EPI0 + NEPI) {
      // ---------------------------------------------------------- loaders
      // per head: the key tile's 2 x 128 rows of 128 bytes as 2,048 16-byte
      // copies, copy i = (key i >> 4, K-block (i >> 3) & 1, chunk i & 7),
      // written where the 128-byte swizzle puts it (chunk ^ (row & 7)); then
      // stage g - 1 is signalled once this thread's copies for it landed.
      // Lane 0 of warp 0 also issues the query tile's two TMA boxes.
      const int lt = (warp == 0 ? 0 : warp < EPI0 ? warp - 1 : warp - (EPI0 + NEPI - 3)) * 32 + lane;
      const int64_t HD = (int64_t)p.Hkv * 128;
      bool ok = true;
      for (int h = 0; h < H && ok; ++h) {
        const uint32_t g = sg + h, s = g % NST;
        if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.empty[s], ((g / NST) & 1) ^ 1, abort, kLimitNs))) {
          ok = false;
          break;
        }
        if (warp == 0 && lane == 0) {
          tc::bar_expect_tx(&sm.full[s], 2 * BBYTES);
          tc::tma_load_2d(sm.b[s][0], &mapQ, h * 128, (int)(t0 + j0), &sm.full[s]);
          tc::tma_load_2d(sm.b[s][1], &mapQ, h * 128 + 64, (int)(t0 + j0), &sm.full[s]);
        }
        const __nv_bfloat16* kh = p.K + (int64_t)(h / kv_group) * 128;
        for (int i = lt; i < 2 * KR * 8; i += NLOAD) {
          const int r = i >> 4, kb = (i >> 3) & 1, ch = i & 7;
          tc::cp_async16(sm.a[s][kb] + r * 128 + ((ch ^ (r & 7)) << 4), kh + sm.kidx[r] * HD + kb * 64 + ch * 8, 16);
        }
        cp_async_commit();
        if (h > 0) {
          cp_async_wait<1>();
          tc::fence_proxy_async();
          tc::bar_arrive(&sm.full[(g - 1) % NST]);
        }
      }
      cp_async_wait<0>();  // on a timeout too: no copy may land after the CTA ends
      if (ok) {
        tc::fence_proxy_async();
        tc::bar_arrive(&sm.full[(sg + H - 1) % NST]);
      }
      if (!ok && lane == 0) {
        sm.abort = 1;
        set_status(p.status, OCCAM_ERR_TIMEOUT);
      }
    } else if (warp == 1) {
      // ---------------------------------------------------------- MMA issuer
      if (lane == 0) {
        const uint32_t idesc = tc::idesc_bf16(KR, TR);
        bool ok = true;
        for (int h = 0; h < H && ok; ++h) {
          const uint32_t g = sg + h, s = g % NST, db = g & 1;
          ok = tc::bar_wait(&sm.full[s], (g / NST) & 1, abort, kLimitNs);
          if (ok && g >= 2) ok = tc::bar_wait(&sm.dfree[db], ((g - 2) >> 1) & 1, abort, kLimitNs);
          if (!ok) break;
          tc::fence_proxy_async();
          tc::fence_after();
#pragma unroll
          for (int kb = 0; kb < 2; ++kb)
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc::mma_bf16(tmem + db * TR, tc::sdesc_sw128(tc::su32(sm.a[s][kb]) + kk * 32),
                           tc::sdesc_sw128(tc::su32(sm.b[s][kb]) + kk * 32), idesc, (kb | kk) ? 1u : 0u);
          tc::mma_commit(&sm.dfull[db]);
          tc::mma_commit(&sm.empty[s]);
        }
        if (!ok) {
          sm.abort = 1;
          set_status(p.status, OCCAM_ERR_TIMEOUT);
        }
      }
      __syncwarp();
    } else if (warp >= EPI0) {  // warps EPI0 .. EPI0 + NEPI - 1
      // ---------------------------------------------------------- softmax warps
      const int ew = warp - EPI0, quad = warp & 3, half = ew >> 2;
      const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
      float acc[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) acc[i] = 0.f;
      bool ok = true;
      for (int h = 0; h < H && ok; ++h) {
        const uint32_t g = sg + h, db = g & 1;
        if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.dfull[db], (g >> 1) & 1, abort, kLimitNs))) {
          ok = false;
          break;
        }
        tc::fence_after();
        uint32_t v[32];
        tc::tmem_ld32(tmem + lane_base + db * TR + half * 32, v);
        ld_wait32(v);
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float2 st = sm.sst[half * 32 + i][h];
          acc[i] = fmaf(tc::ex2(fmaf(__uint_as_float(v[i]), c, -st.x)), st.y, acc[i]);
        }
        tc::fence_before();
        __syncwarp();
        if (lane == 0) tc::bar_arrive(&sm.dfree[db]);
      }
      if (!ok && lane == 0) {
        sm.abort = 1;
        set_status(p.status, OCCAM_ERR_TIMEOUT);
      }
      // the key's max over this warp's text rows and its sum over them (rows
      // past the text contribute 0: their statistics give exp2(-inf) * 0)
      float cmax = 0.f, rs = 0.f;
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        cmax = fmaxf(cmax, acc[i]);
        rs += acc[i];
      }
      sm.part[half][quad][lane] = make_float2(cmax, rs);
    }
    __syncthreads();
    // ---- item end: one thread per key (threads 0..127 = warps 0..3)
    const bool done_ok = !*abort;
    if (tid < KR) {
      const float2 a0 = sm.part[0][tid >> 5][tid & 31], a1 = sm.part[1][tid >> 5][tid & 31];
      float rc = 0.f;
      if (done_ok && tid < nk) {
        if (sm.kreg[tid]) {
          rc = (a0.y + a1.y) * invH;
        } else {
          atomicMax(reinterpret_cast<int*>(&p.s2[sm.kidx[tid]]), __float_as_int(fmaxf(a0.x, a1.x) * invH));
        }
      }
      rc = warp_sum(rc);
      if (lane == 0) sm.rsum[warp] = rc;
    }
    __syncthreads();
    if (tid == 0) {
      sm.last = 0;
      if (done_ok) {
        p.refpart[slot] = (sm.rsum[0] + sm.rsum[1]) + (sm.rsum[2] + sm.rsum[3]);
        __threadfence();
        const int nslots = p.slot_off[b + 1] - p.slot_off[b];
        sm.last = atomicAdd(&p.done[b], 1) == nslots - 1;
      }
    }
    __syncthreads();
    if (sm.last && tid < 32) {
      // the sample's last partial: ref2 = (sum of the partials) / (R M),
      // lane l taking slots l, l + 32, ... in order, then a fixed tree
      __threadfence();
      float acc = 0.f;
      for (int i = p.slot_off[b] + tid; i < p.slot_off[b + 1]; i += 32) acc += __ldcg(&p.refpart[i]);
      acc = warp_sum(acc);
      if (tid == 0) {
        const int R = p.bt.reg_off[p.bt.seg_first[b + 1]] - p.bt.reg_off[p.bt.seg_first[b]];
        const float r2 = (R > 0 && M > 0) ? acc / ((float)R * (float)M) : 0.f;
        p.ref2[b] = r2;
        p.tau2[b] = p.lambda2 * r2;
      }
    }
    __syncthreads();
    sg += H;
  }
  tc::fence_before();
  __syncthreads();
  if (*abort && tid == 0) {
    // let the TMA copies still in flight land before the shared memory goes away
    const uint64_t t0 = tc::globaltimer();
    while (tc::globaltimer() - t0 < 100000ull) {
    }
  }
  __syncthreads();
  tc::fence_after();
  if (warp == 1) tc::tmem_dealloc(tmem, 2 * TR);
}

int launch_scores_tc(const Stage2Params& p, const CUtensorMap& mq64, int grid, cudaStream_t st) {
  const int smem = s2_scores_tc_smem_bytes();
  cudaFuncSetAttribute(s2_scores_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  s2_scores_tc_kernel<<<grid, s2t::THREADS, smem, st>>>(mq64, p);
  count_launch();
  return cudaGetLastError() == cudaSuccess ? 0 : 1;
}

}  // namespace occam
