// stage2.cu -- Stage II of OccamToken (Sec. 3.5): text-to-vision scores at
// LLM layer l. For sample b and text token j, per head h, the softmax runs
// over the S1 rows of b (visual survivors and registers) and the text keys
// 0..j; p[j, v] is the per-head probability averaged over heads;
// s2(v) = max_j p[j, v], s2(r) = mean over registers and over j (Eq. 7;
// App. A, Eqs. 15-16), and tau2 = lambda2 * s2(r) (Eq. 8).
//
// Samples the fused kernel cannot hold take two passes, so that any S1 size
// and any text length fit:
//   stats  (item = sample, 128 text rows, 4 heads, key range): per (j, h)
//          the softmax max and sum over the range's keys; a sample's keys
//          are split into up to 16 ranges so that large samples still
//          spread over the SMs (this file);
//   scores (item = sample, 64 text rows, 128 S1 keys): stage2_scores_tc.cu.
//
// The statistics pass on the 5th-generation tensor cores. Per head of an
// item, the 128 text queries are the MMA's A operand (one text row per TMEM
// lane, two TMA boxes of 128 rows), and the range's keys come as B in blocks
// of 128 (S1 rows of K2 by the S1 list, then the tile's text keys;
// zero-filled past the range), copied by seven loader warps with 16-byte
// cp.async into the 128-byte-swizzled K-major layout. D = Q K^T (128 x 128
// fp32) alternates between two TMEM buffers. Eight epilogue warps (the four
// TMEM lane quadrants, two column halves each) keep an online max and sum
// per text row over their columns, in log2 units; at the head's last block
// the second half hands its pair to the first through shared memory, and
// the first writes the merged partial.
// Roles (512 threads): warps 0, 2, 3 and 12-15 load keys (warp 0 also
// issues the query tile's TMA boxes), warp 1 issues the MMAs, warps 4-11
// are the epilogue. Every wait is bounded; on a timeout the CTA records
// OCCAM_ERR_TIMEOUT, lets its copies land, frees TMEM and returns.
#include "common.cuh"
#include "kernels.cuh"
#include "tc5.cuh"

namespace occam {

namespace s2s {
constexpr int QR = kStatsTile;            // MMA M: the item's text rows
constexpr int KB = 128;                   // keys per block (MMA N)
constexpr int QBYTES = QR * 128;          // one 64-dim K-block of the query operand
constexpr int KBYTES = KB * 128;          // one 64-dim K-block of the key block
constexpr int NST = 3;                    // key block stages
constexpr int NLOAD = 7 * 32;             // key loader threads (warps 0, 2, 3, 12-15)
constexpr int NEPI = 8;                   // epilogue warps (4-11)
constexpr int THREADS = 16 * 32;
constexpr int KT = 64;                    // keys per range chunk (ranges are whole chunks)
constexpr uint64_t kLimitNs = 2000000000ull;
static_assert(kStatsTile == 128, "one text row per TMEM lane");

struct Smem {
  uint8_t q[2][2][QBYTES];   // query tile per head: [buffer][K-block], 128-byte swizzled rows
  uint8_t k[NST][2][KBYTES]; // key block: [stage][K-block]
  float2 part[2][QR];        // the second column half's (max, sum) per text row, by head parity
  uint64_t qfull[2], qempty[2], kfull[NST], kempty[NST], dfull[2], dfree[2], hsync[2];
  uint32_t tmem_base;
  int abort;
};
}  // namespace s2s

int s2_stats_smem_bytes() { return (int)sizeof(s2s::Smem) + 1024; }
static_assert(sizeof(s2s::Smem) + 1024 <= 227 * 1024, "shared memory per CTA");

namespace {

// The sample whose items [off[b], off[b + 1]) hold item it (off ascending).
__device__ __forceinline__ int stats_item_sample(const int32_t* off, int B, int it) {
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (off[mid] <= it) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// One statistics item, decoded the same way by every role.
struct StatsItem {
  int b, M, n_img, total, j0, nq, sp, h_lo, nh, k_lo, k_hi, nb;
  int64_t t0, rbase;
};

__device__ __forceinline__ StatsItem decode_stats_item(const Stage2Params& p, int it) {
  using s2s::KB;
  using s2s::KT;
  StatsItem s;
  s.b = stats_item_sample(p.itemA_off, p.bt.B, it);
  s.t0 = p.bt.text_off[s.b];
  s.M = (int)(p.bt.text_off[s.b + 1] - s.t0);
  s.n_img = p.n1[s.b];
  s.rbase = p.bt.row_off[s.b];
  const int nhg = (p.H + kHeadGroup - 1) / kHeadGroup;
  const int nsp = s2_stat_splits(s.n_img, s.M);
  const int i = it - p.itemA_off[s.b];
  s.j0 = (i / (nhg * nsp)) * kStatsTile;
  const int hg = (i / nsp) % nhg;
  s.sp = i % nsp;
  s.nq = min(kStatsTile, s.M - s.j0);
  const int n_txt = p.Kt ? min(s.j0 + kStatsTile, s.M) : 0;
  s.total = s.n_img + n_txt;
  // the range's chunks [c0, c1) of the tile's key list (may be empty)
  const int nchunks = (s.total + KT - 1) / KT;
  const int per = (nchunks + nsp - 1) / nsp;
  const int c0 = min(nchunks, s.sp * per), c1 = min(nchunks, c0 + per);
  s.k_lo = c0 * KT;
  s.k_hi = min(c1 * KT, s.total);
  s.nb = c0 < c1 ? (s.k_hi - s.k_lo + KB - 1) / KB : 0;
  s.h_lo = hg * kHeadGroup;
  s.nh = min(p.H, s.h_lo + kHeadGroup) - s.h_lo;
  return s;
}

__device__ __forceinline__ void stats_ld_wait(uint32_t (&v)[32]) {
  tc::tmem_wait_ld();
  asm volatile(""
               : "+r"(v[0]), "+r"(v[1]), "+r"(v[2]), "+r"(v[3]), "+r"(v[4]), "+r"(v[5]), "+r"(v[6]), "+r"(v[7]),
                 "+r"(v[8]), "+r"(v[9]), "+r"(v[10]), "+r"(v[11]), "+r"(v[12]), "+r"(v[13]), "+r"(v[14]), "+r"(v[15]),
                 "+r"(v[16]), "+r"(v[17]), "+r"(v[18]), "+r"(v[19]), "+r"(v[20]), "+r"(v[21]), "+r"(v[22]), "+r"(v[23]),
                 "+r"(v[24]), "+r"(v[25]), "+r"(v[26]), "+r"(v[27]), "+r"(v[28]), "+r"(v[29]), "+r"(v[30]), "+r"(v[31]));
}

// Online softmax statistics (log2 units): fold 32 logits x (-inf = masked)
// into (m, z).
__device__ __forceinline__ void fold32(float& m, float& z, const float (&x)[32]) {
  float bm = -INFINITY;
#pragma unroll
  for (int i = 0; i < 32; ++i) bm = fmaxf(bm, x[i]);
  const float mn = fmaxf(m, bm);
  if (mn == -INFINITY) return;
  float acc = 0.f;
#pragma unroll
  for (int i = 0; i < 32; ++i) acc += exp2f(x[i] - mn);
  z = (m == -INFINITY ? 0.f : z * exp2f(m - mn)) + acc;
  m = mn;
}

}  // namespace

__global__ void __launch_bounds__(s2s::THREADS, 1)
    s2_stats_tc_kernel(const __grid_constant__ CUtensorMap mapQ, Stage2Params p) {
  using namespace s2s;
  extern __shared__ unsigned char smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nA = p.counters[CNT_NA];
  if ((int)blockIdx.x >= nA) return;  // no item for this CTA: leave before touching TMEM
  const int H = p.H;
  const int kv_group = p.H / p.Hkv;
  const float c = p.scale * 1.4426950408889634f;
  volatile int* abort = &sm.abort;

  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      tc::bar_init(&sm.qfull[i], 1);
      tc::bar_init(&sm.qempty[i], 1);
      tc::bar_init(&sm.dfull[i], 1);
      tc::bar_init(&sm.dfree[i], NEPI);
      tc::bar_init(&sm.hsync[i], NEPI / 2);
    }
    for (int i = 0; i < NST; ++i) {
      tc::bar_init(&sm.kfull[i], NLOAD);
      tc::bar_init(&sm.kempty[i], 1);
    }
    sm.abort = 0;
    tc::bar_fence_init();
    tc::prefetch_map(&mapQ);
  }
  if (warp == 1) tc::tmem_alloc(&sm.tmem_base, 2 * KB);
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  const uint32_t tmem = sm.tmem_base;

  if (warp == 0 || warp == 2 || warp == 3 || warp >= 12) {
    // ------------------------------------------------------------ loaders
    // block g: 2,048 16-byte copies, copy i = (key i >> 4, K-block
    // (i >> 3) & 1, chunk i & 7) at chunk ^ (key & 7) of its 128-byte row;
    // block g - 1 is signalled once this thread's copies for it landed
    const int lt = (warp == 0 ? 0 : warp < 12 ? warp - 1 : warp - 9) * 32 + lane;
    const int64_t HD = (int64_t)p.Hkv * 128;
    uint32_t g = 0, gq = 0;
    bool ok = true, pending = false;
    for (int it = blockIdx.x; it < nA && ok; it += gridDim.x) {
      const StatsItem s = decode_stats_item(p, it);
      if (s.nb == 0) continue;
      for (int hh = 0; hh < s.nh && ok; ++hh, ++gq) {
        const int h = s.h_lo + hh;
        const int64_t hoff = (int64_t)(h / kv_group) * 128;
        for (int blk = 0; blk < s.nb; ++blk, ++g) {
          const uint32_t st = g % NST;
          if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.kempty[st], ((g / NST) & 1) ^ 1, abort, kLimitNs))) {
            ok = false;
            break;
          }
          if (warp == 0 && blk == 0) {
            const uint32_t qb = gq & 1;
            if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.qempty[qb], ((gq >> 1) & 1) ^ 1, abort, kLimitNs))) {
              ok = false;
              break;
            }
            if (lane == 0) {
              tc::bar_expect_tx(&sm.qfull[qb], 2 * QBYTES);
              tc::tma_load_2d(sm.q[qb][0], &mapQ, h * 128, (int)(s.t0 + s.j0), &sm.qfull[qb]);
              tc::tma_load_2d(sm.q[qb][1], &mapQ, h * 128 + 64, (int)(s.t0 + s.j0), &sm.qfull[qb]);
            }
          }
          const int kb0 = s.k_lo + blk * KB;
          for (int i = lt; i < 2 * KB * 8; i += NLOAD) {
            const int r = i >> 4, kb = (i >> 3) & 1, ch = i & 7;
            const int kk = kb0 + r;
            const __nv_bfloat16* src = p.K;
            int bytes = 0;
            if (kk < s.k_hi) {
              bytes = 16;
              if (kk < s.n_img) {
                const int64_t row = p.dense[s.rbase + kk];
                src = p.K + (in_bounds(row >= 0 && row < p.bt.total_rows, p.status, kSiteTwoPassKeyRow) ? row : 0) * HD;
              } else {
                src = p.Kt + (s.t0 + (kk - s.n_img)) * HD;
              }
              src += hoff + kb * 64 + ch * 8;
            }
            tc::cp_async16(sm.k[st][kb] + r * 128 + ((ch ^ (r & 7)) << 4), src, bytes);
          }
          cp_async_commit();
          if (pending) {
            cp_async_wait<1>();
            tc::fence_proxy_async();
            tc::bar_arrive(&sm.kfull[(g - 1) % NST]);
          }
          pending = true;
        }
      }
    }
    cp_async_wait<0>();  // on a timeout too: no copy may land after the CTA ends
    if (ok && pending) {
      tc::fence_proxy_async();
      tc::bar_arrive(&sm.kfull[(g - 1) % NST]);
    }
    if (!ok && lane == 0) {
      sm.abort = 1;
      set_status(p.status, OCCAM_ERR_TIMEOUT);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t idesc = tc::idesc_bf16(QR, KB);
      uint32_t g = 0, gq = 0;
      bool ok = true;
      for (int it = blockIdx.x; it < nA && ok; it += gridDim.x) {
        const StatsItem s = decode_stats_item(p, it);
        if (s.nb == 0) continue;
        for (int hh = 0; hh < s.nh && ok; ++hh, ++gq) {
          const uint32_t qb = gq & 1;
          ok = tc::bar_wait(&sm.qfull[qb], (gq >> 1) & 1, abort, kLimitNs);
          for (int blk = 0; blk < s.nb && ok; ++blk, ++g) {
            const uint32_t st = g % NST, db = g & 1;
            ok = tc::bar_wait(&sm.kfull[st], (g / NST) & 1, abort, kLimitNs);
            if (ok && g >= 2) ok = tc::bar_wait(&sm.dfree[db], ((g - 2) >> 1) & 1, abort, kLimitNs);
            if (!ok) break;
            tc::fence_proxy_async();
            tc::fence_after();
#pragma unroll
            for (int kb = 0; kb < 2; ++kb)
#pragma unroll
              for (int kk = 0; kk < 4; ++kk)
                tc::mma_bf16(tmem + db * KB, tc::sdesc_sw128(tc::su32(sm.q[qb][kb]) + kk * 32),
                             tc::sdesc_sw128(tc::su32(sm.k[st][kb]) + kk * 32), idesc, (kb | kk) ? 1u : 0u);
            tc::mma_commit(&sm.dfull[db]);
            tc::mma_commit(&sm.kempty[st]);
          }
          if (ok) tc::mma_commit(&sm.qempty[qb]);  // the head's query tile is read
        }
      }
      if (!ok) {
        sm.abort = 1;
        set_status(p.status, OCCAM_ERR_TIMEOUT);
      }
    }
    __syncwarp();
  } else if (warp >= 4 && warp < 4 + NEPI) {
    // ------------------------------------------------------------ epilogue
    const int quad = warp & 3, half = (warp - 4) >> 2;  // text rows quad * 32 + lane, columns half * 64 ..
    const int row = quad * 32 + lane;
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    uint32_t g = 0, gq = 0;
    bool ok = true;
    for (int it = blockIdx.x; it < nA && ok; it += gridDim.x) {
      const StatsItem s = decode_stats_item(p, it);
      const int j = s.j0 + row;
      if (s.nb == 0) {  // an empty key range: neutral partials
        if (half == 0 && row < s.nq)
          for (int hh = 0; hh < s.nh; ++hh)
            p.stats[((s.t0 + j) * H + s.h_lo + hh) * kStatSplits + s.sp] = make_float2(-INFINITY, 0.f);
        continue;
      }
      for (int hh = 0; hh < s.nh && ok; ++hh, ++gq) {
        float m = -INFINITY, z = 0.f;
        for (int blk = 0; blk < s.nb; ++blk, ++g) {
          const uint32_t db = g & 1;
          if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.dfull[db], (g >> 1) & 1, abort, kLimitNs))) {
            ok = false;
            break;
          }
          tc::fence_after();
#pragma unroll
          for (int q = 0; q < 2; ++q) {
            uint32_t v[32];
            tc::tmem_ld32(tmem + lane_base + db * KB + half * 64 + q * 32, v);
            stats_ld_wait(v);
            const int kc = s.k_lo + blk * KB + half * 64 + q * 32;
            float x[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int kk = kc + i;
              const bool valid = kk < s.k_hi && (kk < s.n_img || kk - s.n_img <= j);
              x[i] = valid ? __uint_as_float(v[i]) * c : -INFINITY;
            }
            fold32(m, z, x);
          }
          if (blk == s.nb - 1) {
            // the head's last block: the second half hands (m, z) to the first
            const uint32_t hp = gq & 1;
            if (half == 1) {
              sm.part[hp][row] = make_float2(m, z);
              __syncwarp();
              if (lane == 0) tc::bar_arrive(&sm.hsync[hp]);
            } else {
              if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.hsync[hp], (gq >> 1) & 1, abort, kLimitNs))) {
                ok = false;
                break;
              }
              const float2 o = sm.part[hp][row];
              const float mx = fmaxf(m, o.x);
              float zz = 0.f;
              if (mx != -INFINITY)
                zz = (m == -INFINITY ? 0.f : z * exp2f(m - mx)) + (o.x == -INFINITY ? 0.f : o.y * exp2f(o.x - mx));
              if (row < s.nq) p.stats[((s.t0 + j) * H + s.h_lo + hh) * kStatSplits + s.sp] = make_float2(mx, zz);
            }
          }
          // D[db] is free once every epilogue warp read it (for the first
          // half, also its partner's pair: that keeps part[] single-writer)
          tc::fence_before();
          __syncwarp();
          if (lane == 0) tc::bar_arrive(&sm.dfree[db]);
        }
      }
    }
    if (!ok && lane == 0) {
      sm.abort = 1;
      set_status(p.status, OCCAM_ERR_TIMEOUT);
    }
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
  if (warp == 1) tc::tmem_dealloc(tmem, 2 * KB);
}

int launch_stats_tc(const Stage2Params& p, const CUtensorMap& mq128, int grid, cudaStream_t st) {
  cudaFuncSetAttribute(s2_stats_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, s2_stats_smem_bytes());
  s2_stats_tc_kernel<<<grid, s2s::THREADS, s2_stats_smem_bytes(), st>>>(mq128, p);
  count_launch();
  return cudaGetLastError() == cudaSuccess ? 0 : 1;
}

}  // namespace occam
