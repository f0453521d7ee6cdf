// stage1_tc.cu -- mutual Stage-I scoring on the 5th-generation tensor cores
// (tcgen05 + TMEM + TMA).
//
// What it computes (Sec. 3.4, Eq. 6; App. A, Eq. 13): in segment s with n
// rows, every row u attends to every row v per head h with
// A_h(u -> v) = softmax_v(q_{u,h} k_{v,h} / sqrt(d1)), and
// s1[v] = 1/n sum_u 1/H sum_h A_h(u -> v).
// Two launches of one kernel template:
//   pass 1: per (segment, tile of 128 query rows, head) the query rows'
//           softmax log-sums L[h][u] = log2 sum_v exp2(c q_u k_v), with
//           c = log2(e) / sqrt(d1), over all the segment's keys (stored
//           negated, as the second pass adds them);
//   pass 2: per (segment, tile of 128 key rows, group of 4 heads) the
//           attention each key receives, sum_h sum_u exp2(c q_u k_v - L[h][u]),
//           over the group's heads and all query rows; a small third kernel
//           sums the groups' shares in order into s1.
// In both, the CTA's 128 tile rows are the TMEM lanes (the MMA's A operand)
// and the other side streams in blocks of 256 rows (the B operand):
// S = A B^T is 128 x 256 fp32 in TMEM, from 4-5 tcgen05.mma of K = 16.
// Q1 and K1 are read as 3-D TMA boxes {64 dims, 1 head, 128 rows} with the
// 128-byte swizzle, plus {16 dims, 1 head, 128 rows} with the 32-byte swizzle
// for dims 64-79; dims past d1 (72 -> 80) come zero-filled by the box, so the
// padded K-step adds nothing.
// Roles (640 threads): warp 0 issues the TMA loads, warp 1 the MMAs, warps
// 4-19 (four per TMEM lane quadrant, each taking 64 of the 256 columns) the
// softmax arithmetic; four warps per SM sub-partition keep the exponential
// unit fed through the load -> max -> exp2 latency chains. A tiles, B blocks and the TMEM accumulator are double
// buffered. Every wait is bounded; on a timeout the CTA records
// OCCAM_ERR_TIMEOUT, lets its copies land, frees TMEM and returns.
#include "common.cuh"
#include "kernels.cuh"
#include "tc5.cuh"

namespace occam {

namespace m1 {
constexpr int AR = 128;                   // tile rows (TMEM lanes)
constexpr int BR = 256;                   // block rows (MMA N)
constexpr int ABYTES = AR * 128;          // K-block 0 (dims 0-63) of an A tile
constexpr int BBYTES = BR * 128;          // K-block 0 of a B block
constexpr int ABYTES1 = AR * 32;          // K-block 1 (dims 64-79, 32-byte rows) of an A tile
constexpr int BBYTES1 = BR * 32;
constexpr int NEPI = 16;                  // softmax warps: NEPI / 4 per TMEM lane quadrant
constexpr int QW = NEPI / 4;              // softmax warps per quadrant
constexpr int COLS = BR / QW;             // accumulator columns per softmax warp (64)
constexpr int EPI0 = 4;                   // first softmax warp
constexpr int THREADS = (EPI0 + NEPI) * 32;
constexpr int NBB = 4;                    // B blocks in flight (a ring; A tiles and accumulators: 2 each)
static_assert(COLS == 64, "one 64-column TMEM load per softmax warp and block");
constexpr uint64_t kLimitNs = 2000000000ull;

// A decoded work item: segment, first row of its tile, first head, the
// segment's rows and its first row in the batch.
struct MutItem {
  int seg, a0, h, n;
  int64_t sb;
};

struct Smem {
  uint8_t a[2][ABYTES];     // K-block 0 per buffer
  uint8_t b[NBB][BBYTES];
  uint8_t a1[2][ABYTES1];   // K-block 1 per buffer
  uint8_t b1[NBB][BBYTES1];
  float lsm[2][NEPI][COLS];  // pass 2: minus the log-sums of each softmax warp's columns (a ring of 2 steps)
  float2 part[2][QW - 1][4][32];  // partials of quarters 1.. per (item parity, quarter, quadrant, lane)
  int32_t item[8];          // the ii-th work item, by ii & 7 (-1: no more)
  MutItem itm[8];           // ... decoded by the TMA producer for every role
  uint64_t afull[2], aempty[2], bfull[NBB], bempty[NBB], dfull[2], dfree[2], hb[2][4], inext[8], mdone;
  uint64_t aready[2], bready[NBB];  // pass 2 with the log-sums folded into the MMA: tiles completed for it
  uint32_t tmem_base;
  int abort;
};
}  // namespace m1

static_assert(sizeof(m1::Smem) + 1024 <= 227 * 1024, "shared memory per CTA");

int mutual_tc_smem_bytes() { return (int)sizeof(m1::Smem) + 1024; }

namespace {

__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, int x, int y, int z, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], "
      "[%5];" ::"r"(tc::su32(dst)),
      "l"(map), "r"(x), "r"(y), "r"(z), "r"(tc::su32(bar))
      : "memory");
}

__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(tc::su32(dst)), "l"(src) : "memory");
}

__device__ __forceinline__ void wait_ld64(uint32_t (&v)[64]) {
  tc::tmem_wait_ld();
  asm volatile("" : OCCAM_TC_RW64(v));
}

}  // namespace

// Work items, taken from a queue by a persistent grid (one CTA per SM):
// PASS 1: (segment, tile of 128 query rows, head), A = query tile, B = key
//         blocks of that head;
// PASS 2: (segment, tile of 128 key rows, group of 4 heads), A = key tile,
//         B = query blocks, for the group's heads in turn.
// The producer thread draws items (skipping tiles past a segment's rows) and
// hands each to the MMA and softmax warps through an 8-deep ring in shared
// memory (the producer runs at most a few steps ahead, so a slot is read
// before it comes round again); buffer and phase counters run on across
// items, so the next item's loads overlap the current item's tail.

template <int PASS>
__device__ __forceinline__ bool mut_item(const MutualTcParams& p, int it, m1::MutItem& w) {
  const int sub_n = PASS == 1 ? p.H : p.hgroups;  // heads (pass 1) or head groups (pass 2) per tile
  const int per_seg = p.tiles * sub_n;
  w.seg = it / per_seg;
  const int rem = it - w.seg * per_seg;
  const int tile = rem / sub_n;
  w.h = (rem - tile * sub_n) * (PASS == 1 ? 1 : kMutHeadGroup);  // first head of the item
  w.a0 = tile * m1::AR;
  w.sb = p.bt.seg_off[w.seg];
  w.n = (int)(p.bt.seg_off[w.seg + 1] - w.sb);
  return w.a0 < w.n;
}

template <int PASS, bool FOLD>
__global__ void __launch_bounds__(m1::THREADS, 1)
    mutual_tc_kernel(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
                     const __grid_constant__ CUtensorMap mapA1, const __grid_constant__ CUtensorMap mapB1,
                     MutualTcParams p) {
  using namespace m1;
  extern __shared__ unsigned char smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int H = p.H;
  const int total = p.bt.S_tot * p.tiles * (PASS == 1 ? H : p.hgroups);
  const int nkb = p.d1 > 64 ? 2 : 1;         // K-blocks of 64 dims
  const int nks = (p.d1 + 15) / 16;          // K-steps of 16 dims
  int* queue = p.queue + (PASS - 1);
  volatile int* abort = &sm.abort;

  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      tc::bar_init(&sm.afull[i], 1);
      tc::bar_init(&sm.aempty[i], 1);

      tc::bar_init(&sm.dfull[i], 1);
      tc::bar_init(&sm.dfree[i], NEPI);
    }
    for (int i = 0; i < NBB; ++i) {
      tc::bar_init(&sm.bfull[i], 1);
      tc::bar_init(&sm.bempty[i], 1);
      tc::bar_init(&sm.bready[i], 2);
    }
    for (int i = 0; i < 2; ++i) tc::bar_init(&sm.aready[i], 2);
    for (int i = 0; i < 8; ++i) tc::bar_init(&sm.hb[i >> 2][i & 3], QW - 1);
    for (int i = 0; i < 8; ++i) tc::bar_init(&sm.inext[i], 1);
    tc::bar_init(&sm.mdone, 1);
    sm.abort = 0;
    tc::bar_fence_init();
    tc::prefetch_map(&mapA);
    tc::prefetch_map(&mapB);
    tc::prefetch_map(&mapA1);
    tc::prefetch_map(&mapB1);
  }
  if (warp == 1) tc::tmem_alloc(&sm.tmem_base, 512);
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem = sm.tmem_base;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      uint32_t na = 0, nbk = 0;
      for (int ii = 0;; ++ii) {
        int it;
        MutItem w;
        do {
          it = atomicAdd(queue, 1);
        } while (it < total && !mut_item<PASS>(p, it, w));
        if (it < total) sm.itm[ii & 7] = w;
        sm.item[ii & 7] = it < total && !*abort ? it : -1;
        tc::bar_arrive(&sm.inext[ii & 7]);
        if (it >= total || *abort) break;
        const int64_t sb = w.sb;
        const int nb = (w.n + BR - 1) / BR;
        const int nheads = PASS == 1 ? 1 : min(kMutHeadGroup, H - w.h);
        bool ok = true;
        // step s is block jb of head h (counters instead of a division per step)
        for (int s = 0, h = w.h, jb = 0; s < nheads * nb && ok; ++s, jb = jb + 1 == nb ? 0 : jb + 1, h += jb == 0) {
          if (jb == 0) {
            const int ab = na & 1;
            if (!tc::bar_wait(&sm.aempty[ab], ((na >> 1) & 1) ^ 1, abort, kLimitNs)) {
              ok = false;
              break;
            }
            tc::bar_expect_tx(&sm.afull[ab], (uint32_t)(ABYTES + (nkb > 1 ? ABYTES1 : 0)));
            tma_load_3d(sm.a[ab], &mapA, 0, h, (int)(sb + w.a0), &sm.afull[ab]);
            if (nkb > 1) tma_load_3d(sm.a1[ab], &mapA1, 64, h, (int)(sb + w.a0), &sm.afull[ab]);
            ++na;
          }
          const int bb = nbk % NBB;
          if (!tc::bar_wait(&sm.bempty[bb], ((nbk / NBB) & 1) ^ 1, abort, kLimitNs)) {
            ok = false;
            break;
          }
          tc::bar_expect_tx(&sm.bfull[bb], (uint32_t)(BBYTES + (nkb > 1 ? BBYTES1 : 0)));
          for (int hh = 0; hh < BR / AR; ++hh) {
            const int y = (int)(sb + jb * BR + hh * AR);
            tma_load_3d(sm.b[bb] + hh * ABYTES, &mapB, 0, h, y, &sm.bfull[bb]);
            if (nkb > 1) tma_load_3d(sm.b1[bb] + hh * ABYTES1, &mapB1, 64, h, y, &sm.bfull[bb]);
          }
          ++nbk;
        }
        if (!ok) {
          sm.abort = 1;
          set_status(p.status, OCCAM_ERR_TIMEOUT);
          // tell the other roles to stop at the next hand-out
          sm.item[(ii + 1) & 7] = -1;
          tc::bar_arrive(&sm.inext[(ii + 1) & 7]);
          break;
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = tc::idesc_bf16(AR, BR);
      uint32_t na = 0, sg = 0;
      for (int ii = 0;; ++ii) {
        if (!tc::bar_wait(&sm.inext[ii & 7], (ii >> 3) & 1, abort, kLimitNs)) {
          sm.abort = 1;
          set_status(p.status, OCCAM_ERR_TIMEOUT);
          break;
        }
        const int it = *reinterpret_cast<volatile int*>(&sm.item[ii & 7]);
        if (it < 0) break;
        const MutItem w = sm.itm[ii & 7];
        const int nb = (w.n + BR - 1) / BR;
        const int nheads = PASS == 1 ? 1 : min(kMutHeadGroup, H - w.h);
        bool ok = true;
        for (int s = 0, jb = 0; s < nheads * nb; ++s, ++sg, jb = jb + 1 == nb ? 0 : jb + 1) {
          const int ab = na & 1, bb = sg % NBB, db = sg & 1;
          if (jb == 0) ok = tc::bar_wait(FOLD ? &sm.aready[ab] : &sm.afull[ab], (na >> 1) & 1, abort, kLimitNs);
          if (ok) ok = tc::bar_wait(FOLD ? &sm.bready[bb] : &sm.bfull[bb], (sg / NBB) & 1, abort, kLimitNs);
          if (ok && sg >= 2) ok = tc::bar_wait(&sm.dfree[db], ((sg - 2) >> 1) & 1, abort, kLimitNs);
          if (!ok) break;
          tc::fence_after();
          const uint32_t abase = tc::su32(sm.a[ab]), bbase = tc::su32(sm.b[bb]);
          for (int ks = 0; ks < nks && ks < 4; ++ks)
            tc::mma_bf16(tmem + db * BR, tc::sdesc_sw128(abase + ks * 32), tc::sdesc_sw128(bbase + ks * 32), idesc,
                         ks > 0 ? 1u : 0u);
          // dims 64-79: one K-step over the 32-byte rows
          if (nks > 4)
            tc::mma_bf16(tmem + db * BR, tc::sdesc_sw32(tc::su32(sm.a1[ab])), tc::sdesc_sw32(tc::su32(sm.b1[bb])),
                         idesc, 1u);
          tc::mma_commit(&sm.dfull[db]);
          tc::mma_commit(&sm.bempty[bb]);
          if (jb == nb - 1) {
            tc::mma_commit(&sm.aempty[ab]);
            ++na;
          }
        }
        if (!ok) {
          sm.abort = 1;
          set_status(p.status, OCCAM_ERR_TIMEOUT);
          break;
        }
      }
      tc::mma_commit(&sm.mdone);
      if (!tc::bar_wait(&sm.mdone, 0, nullptr, kLimitNs)) set_status(p.status, OCCAM_ERR_TIMEOUT);
    }
    __syncwarp();
  } else if (FOLD && (warp == 2 || warp == 3)) {
    // ------------------------------------------------------------ fold warps
    // Pass 2 with d1 = 72: dims 72-79 of the last K-step arrive zero-filled
    // by the TMA box. Into dims 72-74 go 1.0 on the key side (A) and, on the
    // query side (B), a three-term bf16 split of -L_u / c (each term the
    // rounding of what the previous ones leave, so the three hold 24
    // significant bits), so the MMA yields S - L_u / c and the softmax warps
    // need only c times it. A query row past the segment gets -1e30, whose
    // exponential is 0. In the 32-byte-swizzled rows, dims 72-79 (16-byte
    // chunk 1 of row r) sit in chunk 1 ^ ((r >> 2) & 1). Warp 2 takes the
    // first half of each tile's rows, warp 3 the second.
    const float inv_c = 1.0f / p.scale_log2;
    const int half = warp - 2;
    const int64_t R = p.bt.total_rows;
    uint32_t na = 0, nbk = 0;
    for (int ii = 0;; ++ii) {
      if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.inext[ii & 7], (ii >> 3) & 1, nullptr, kLimitNs))) {
        sm.abort = 1;
        set_status(p.status, OCCAM_ERR_TIMEOUT);
        break;
      }
      const int it = *reinterpret_cast<volatile int*>(&sm.item[ii & 7]);
      if (it < 0) break;
      const MutItem w = sm.itm[ii & 7];
      const int n = w.n;
      const int64_t sb = w.sb;
      const int nb = (n + BR - 1) / BR;
      const int steps = min(kMutHeadGroup, H - w.h) * nb;
      // -L of the block's query rows lane + 32 k, loaded a step ahead
      // (clamped to the segment; rows past it are replaced below)
      constexpr int KR = BR / 64;  // B rows per lane and step
      float lpre[KR];
      auto load_l = [&](int ht, int tb) {  // block tb of head ht
        const int base = tb * BR + half * (BR / 2);
#pragma unroll
        for (int k = 0; k < KR; ++k)
          lpre[k] = __ldcg(&p.lsum[(int64_t)ht * R + sb + min(base + lane + 32 * k, n - 1)]);
      };
      load_l(w.h, 0);
      bool ok = true;
      for (int s = 0, h = w.h, jb = 0; s < steps; ++s, jb = jb + 1 == nb ? 0 : jb + 1, h += jb == 0) {
        if (jb == 0) {
          const int ab = na & 1;
          if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.afull[ab], (na >> 1) & 1, nullptr, kLimitNs))) {
            ok = false;
            break;
          }
          for (int r = half * (AR / 2) + lane; r < (half + 1) * (AR / 2); r += 32)
            *reinterpret_cast<uint4*>(sm.a1[ab] + r * 32 + 16 * (1 ^ ((r >> 2) & 1))) =
                make_uint4(0x3F803F80u, 0x00003F80u, 0u, 0u);  // bf16 1.0 in dims 72, 73, 74
          tc::fence_proxy_async();
          __syncwarp();
          if (lane == 0) tc::bar_arrive(&sm.aready[ab]);
          ++na;
        }
        const int bb = nbk % NBB;
        if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.bfull[bb], (nbk / NBB) & 1, nullptr, kLimitNs))) {
          ok = false;
          break;
        }
        float cur[KR];
#pragma unroll
        for (int k = 0; k < KR; ++k) cur[k] = lpre[k];
        if (s + 1 < steps) {
          if (jb + 1 == nb) load_l(h + 1, 0);
          else load_l(h, jb + 1);
        }
#pragma unroll
        for (int k = 0; k < KR; ++k) {
          const int r = half * (BR / 2) + lane + 32 * k;
          uint4 t4 = make_uint4(__bfloat16_as_ushort(__float2bfloat16_rn(-1e30f)), 0u, 0u, 0u);
          if (jb * BR + r < n) {
            const float y = cur[k] * inv_c;  // -L / c
            const __nv_bfloat16 h1 = __float2bfloat16_rn(y);
            const float r1 = y - __bfloat162float(h1);
            const __nv_bfloat16 h2 = __float2bfloat16_rn(r1);
            const float r2 = r1 - __bfloat162float(h2);
            const __nv_bfloat16 h3 = __float2bfloat16_rn(r2);
            t4.x = (uint32_t)__bfloat16_as_ushort(h1) | ((uint32_t)__bfloat16_as_ushort(h2) << 16);
            t4.y = (uint32_t)__bfloat16_as_ushort(h3);
          }
          *reinterpret_cast<uint4*>(sm.b1[bb] + r * 32 + 16 * (1 ^ ((r >> 2) & 1))) = t4;
        }
        tc::fence_proxy_async();
        __syncwarp();
        if (lane == 0) tc::bar_arrive(&sm.bready[bb]);
        ++nbk;
      }
      if (!ok) {
        sm.abort = 1;
        set_status(p.status, OCCAM_ERR_TIMEOUT);
        break;
      }
    }
  } else if (warp >= EPI0) {
    // ------------------------------------------------------------ softmax warps
    const int ew = warp - EPI0;
    const int quad = warp & 3, qtr = ew >> 2;           // TMEM lane quadrant; which 64 of the 256 columns
    const int row = quad * 32 + lane;                   // tile row = TMEM lane
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    const float c = p.scale_log2;
    const int64_t R = p.bt.total_rows;
    uint32_t sg = 0;
    for (int ii = 0;; ++ii) {
      if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.inext[ii & 7], (ii >> 3) & 1, nullptr, kLimitNs))) {
        sm.abort = 1;
        set_status(p.status, OCCAM_ERR_TIMEOUT);
        break;
      }
      const int it = *reinterpret_cast<volatile int*>(&sm.item[ii & 7]);
      if (it < 0) break;
      const MutItem w = sm.itm[ii & 7];
      const int n = w.n;
      const int64_t sb = w.sb;
      const int nb = (n + BR - 1) / BR;
      const int steps = (PASS == 1 ? 1 : min(kMutHeadGroup, H - w.h)) * nb;
      const bool vrow = w.a0 + row < n;
      const int pp = ii & 1;
      float m = -INFINITY, z = 0.f;  // pass 1: running max / sum (log2 domain)
      float acc = 0.f;               // pass 2: attention received by this key row
      bool ok = true;
      // step s is block jb of head h (counters instead of a division per step)
      for (int s = 0, h = w.h, jb = 0; s < steps; ++s, ++sg, jb = jb + 1 == nb ? 0 : jb + 1, h += jb == 0) {
        const int col0 = jb * BR + qtr * COLS;          // segment-relative index of this warp's column 0
        if (PASS == 2 && !FOLD) {
          // minus the log-sums of this warp's 64 query columns (past the
          // segment: -inf, which contributes 0) come by cp.async into a ring
          // of two step slots, one step ahead; the item's first step's are
          // fetched here. The slot refilled below was last read in the
          // previous step, which every lane of the warp has finished.
          auto fetch = [&](int t, int ht, int tb) {  // step t = block tb of head ht
            const int ct = tb * BR + qtr * COLS;
#pragma unroll
            for (int i = 0; i < 2; ++i) {
              const int qq = ct + lane * 2 + i;
              float* dst = &sm.lsm[t & 1][ew][lane * 2 + i];
              if (qq < n)
                cp_async4(dst, &p.lsum[(int64_t)ht * R + sb + qq]);
              else
                *dst = -INFINITY;
            }
            cp_async_commit();
          };
          if (s == 0) fetch(0, w.h, 0);
          cp_async_wait<0>();
          __syncwarp();
          if (s + 1 < steps) {
            if (jb + 1 == nb) fetch(s + 1, h + 1, 0);
            else fetch(s + 1, h, jb + 1);
          }
        }
        const int db = sg & 1;
        if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.dfull[db], (sg >> 1) & 1, nullptr, kLimitNs))) {
          ok = false;
          break;
        }
        tc::fence_after();
        {
          uint32_t v[64];
          tc::tmem_ld64(tmem + lane_base + db * BR + qtr * COLS, v);
          wait_ld64(v);
          if (PASS == 1) {
            // keys past the segment are masked out of this row's softmax
            const int lim = n - col0;
            if (lim < 64) {
#pragma unroll
              for (int i = 0; i < 64; ++i) v[i] = i < lim ? v[i] : 0xff800000u;  // -inf
            }
            // max as a tree of three-input maxima (32 operations for 64
            // values; short dependency chains)
            float t[22];
#pragma unroll
            for (int i = 0; i < 21; ++i)
              t[i] = tc::fmax3(__uint_as_float(v[3 * i]), __uint_as_float(v[3 * i + 1]), __uint_as_float(v[3 * i + 2]));
            t[21] = __uint_as_float(v[63]);
            float u[8];
#pragma unroll
            for (int i = 0; i < 7; ++i) u[i] = tc::fmax3(t[3 * i], t[3 * i + 1], t[3 * i + 2]);
            u[7] = t[21];
            // c > 0: the max of c l is c times the max of l
            const float mx = fmaxf(tc::fmax3(u[0], u[1], u[2]), tc::fmax3(u[3], u[4], fmaxf(u[5], fmaxf(u[6], u[7])))) * c;
            if (mx != -INFINITY) {
              const float2 cc = make_float2(c, c), om = make_float2(-mx, -mx);
              float2 ap[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                float2 x = __ffma2_rn(make_float2(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1])), cc, om);
                x.x = tc::ex2(x.x);
                x.y = tc::ex2(x.y);
                ap[i & 3] = __fadd2_rn(ap[i & 3], x);
              }
              const float2 a2 = __fadd2_rn(__fadd2_rn(ap[0], ap[1]), __fadd2_rn(ap[2], ap[3]));
              const float a = a2.x + a2.y;
              const bool up = mx > m;
              const float e = tc::ex2(up ? m - mx : mx - m);
              z = up ? fmaf(z, e, a) : fmaf(a, e, z);
              m = fmaxf(m, mx);
            }
          } else {
            const float2* nl = reinterpret_cast<const float2*>(sm.lsm[s & 1][ew]);
            const float2 cc = make_float2(c, c);
            float2 ap[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              // FOLD: the accumulator already holds S - L / c
              const float2 sv = make_float2(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1]));
              float2 x = FOLD ? __fmul2_rn(sv, cc) : __ffma2_rn(sv, cc, nl[i]);
              x.x = tc::ex2(x.x);
              x.y = tc::ex2(x.y);
              ap[i & 3] = __fadd2_rn(ap[i & 3], x);
            }
            const float2 a2 = __fadd2_rn(__fadd2_rn(ap[0], ap[1]), __fadd2_rn(ap[2], ap[3]));
            acc += a2.x + a2.y;
          }
        }
        tc::fence_before();
        __syncwarp();
        const bool last = s == steps - 1;
        if (qtr > 0 && last) {
          // quarters 1.. hand their partials to quarter 0
          sm.part[pp][qtr - 1][quad][lane] = make_float2(PASS == 1 ? m : acc, z);
          __syncwarp();
          if (lane == 0) tc::bar_arrive(&sm.hb[pp][quad]);
        }
        if (qtr == 0 && last) {
          // read the partners' partials before releasing this step's
          // accumulator: their next writes to the slots wait on that release
          if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.hb[pp][quad], (ii >> 1) & 1, nullptr, kLimitNs))) {
            ok = false;
            break;
          }
          if (PASS == 1) {
#pragma unroll
            for (int q = 0; q < QW - 1; ++q) {
              const float2 o = sm.part[pp][q][quad][lane];
              if (o.x != -INFINITY) {
                const bool up = o.x > m;
                const float e = tc::ex2(up ? m - o.x : o.x - m);
                z = up ? fmaf(z, e, o.y) : fmaf(o.y, e, z);
                m = fmaxf(m, o.x);
              }
            }
            // -L, L = log2 of the row's sum of exp2(c q k) over the segment's keys
            if (vrow && in_bounds(sb + w.a0 + row < R, p.status, kSiteMutualRow))
              p.lsum[(int64_t)w.h * R + sb + w.a0 + row] = -(m + log2f(z));
          } else {
            float tot = acc;
#pragma unroll
            for (int q = 0; q < QW - 1; ++q) tot += sm.part[pp][q][quad][lane].x;
            // this head group's share of s1 (summed over the groups in order afterwards)
            if (vrow && in_bounds(sb + w.a0 + row < R, p.status, kSiteMutualRow))
              p.part[(int64_t)(w.h / kMutHeadGroup) * R + sb + w.a0 + row] = tot * p.inv_h / (float)n;
          }
          __syncwarp();
        }
        if (lane == 0) tc::bar_arrive(&sm.dfree[db]);
      }
      if (!ok) {
        sm.abort = 1;
        set_status(p.status, OCCAM_ERR_TIMEOUT);
        break;
      }
    }
  }

  // ------------------------------------------------------------ teardown
  tc::fence_before();
  __syncthreads();
  if (sm.abort && tid == 0) {
    // let the TMA copies still in flight land before the CTA's shared memory goes away
    const uint64_t t0 = tc::globaltimer();
    while (tc::globaltimer() - t0 < 100000ull) {
    }
  }
  __syncthreads();
  tc::fence_after();
  if (warp == 1) tc::tmem_dealloc(tmem, 512);
}

// s1 = the sum of the head groups' shares, in group order (deterministic)
__global__ void __launch_bounds__(256) mutual_reduce_kernel(MutualTcParams p) {
  const int64_t R = p.bt.total_rows;
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < R; r += (int64_t)gridDim.x * blockDim.x) {
    float v = 0.f;
    for (int g = 0; g < p.hgroups; ++g) v += __ldcg(&p.part[(int64_t)g * R + r]);
    p.s1[r] = v;
    if (p.s2_zero) p.s2_zero[r] = 0.f;
  }
  pdl_trigger();  // the finalize kernel may start its input-only prologue
}

void launch_mutual_tc(const MutualTcParams& p, const CUtensorMap& mq, const CUtensorMap& mk, const CUtensorMap& mq1,
                      const CUtensorMap& mk1, int sms, cudaStream_t st) {
  const int smem = mutual_tc_smem_bytes();
  cudaFuncSetAttribute(mutual_tc_kernel<1, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  cudaFuncSetAttribute(mutual_tc_kernel<2, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  cudaFuncSetAttribute(mutual_tc_kernel<2, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  mutual_tc_kernel<1, false><<<sms, m1::THREADS, smem, st>>>(mq, mk, mq1, mk1, p);
  // with d1 = 72 the last K-step has free dims for the log-sums (see the fold warp)
  if (p.d1 == 72)
    mutual_tc_kernel<2, true><<<sms, m1::THREADS, smem, st>>>(mk, mq, mk1, mq1, p);
  else
    mutual_tc_kernel<2, false><<<sms, m1::THREADS, smem, st>>>(mk, mq, mk1, mq1, p);
  mutual_reduce_kernel<<<sms * 2, 256, 0, st>>>(p);
  count_launch(3);
}

}  // namespace occam
