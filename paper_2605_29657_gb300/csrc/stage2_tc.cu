// stage2_tc.cu -- fused Stage-II scoring on the 5th-generation tensor cores
// (tcgen05 + TMEM), for samples whose S1 fits a 4-CTA cluster.
//
// What it computes (Sec. 3.5, Eq. 7; App. A, Eqs. 15-16): for sample b, text
// token j and head h, A_{j,h} = softmax over {S1 rows of b} u {text keys 0..j}
// of q_{j,h} k^T / sqrt(d2); P[j, v] = sum_h A_{j,h}(v); s2(v) = max_j P[j, v] / H
// for visual S1 rows and the registers' sum_j P[j, r] / H for s2(r).
//
// Work item = (sample, tile of 128 text rows), processed by one cluster of 4
// CTAs. The text rows are the 128 TMEM lanes; each CTA owns a quarter of the
// sample's S1 keys and of the causal text keys. Per head:
//   1. three producer warps stream the CTA's key rows in 64-key chunks with
//      16-byte cp.async into the 128-byte-swizzled operand layout (S1 rows
//      are gathered by index straight from K2: pruned rows are never read),
//      and the head's 128 x 128 query tile arrives by TMA;
//   2. the MMA warp computes S = Q K^T per chunk into a TMEM buffer;
//   3. eight epilogue warps (two per TMEM lane quadrant, one thread per text
//      row, taking alternate chunks) keep the row's running softmax max / sum
//      over their chunks, then exchange them with every epilogue warp of the
//      cluster through distributed shared memory, so every CTA holds the
//      exact per-row max and sum over all keys of the head;
//   4. the image chunks are multiplied again (S is recomputed from shared
//      memory) and exp(l - max) / sum is accumulated into the head-summed
//      probabilities P, which live in TMEM for the whole item.
// After the last head every CTA reduces its P columns over the valid rows:
// column max -> s2 (atomicMax on the fp32 bit pattern, exact and order-free
// since P >= 0), register columns -> a partial of s2(r) reduced in fixed order.
// Each key row of K2 is read from HBM once per text tile; the second pass
// over a head's chunks hits L2.
#include "common.cuh"
#include "kernels.cuh"
#include "tc5.cuh"

namespace occam {

namespace s2f {
constexpr int C = kFusedCluster;       // CTAs per cluster
constexpr int QR = 128;                // text rows per item (TMEM lanes)
constexpr int KC = 64;                 // keys per chunk (MMA N)
constexpr int NST = 4;                 // key-chunk ring stages
constexpr int PMAX = kFusedMaxOwnImg;  // max S1 keys per CTA (P columns)
constexpr int TMAX = kFusedMaxOwnTxt;  // max text keys per CTA
constexpr int QBYTES = QR * 256;       // one head's query tile: 2 K-blocks x 128 rows x 128 B
constexpr int KBYTES = KC * 256;       // one chunk: 2 K-blocks x 64 rows x 128 B
constexpr int NPROD = 3;               // producer warps (0-2); warp 3 issues MMAs; then the epilogue warps
constexpr int MMA_WARP = NPROD;
constexpr int EPI_WARP0 = NPROD + 1;
constexpr int NEPI = kFusedEpiWarps;   // two per TMEM lane quadrant; half h takes chunks with (index & 1) == h
constexpr int THREADS = (NPROD + 1 + NEPI) * 32;
constexpr uint32_t IDESC = tc::idesc_bf16(128, KC);
constexpr uint32_t TMEM_COLS = 512;
constexpr int S_COL = 0;               // two S buffers of KC columns
constexpr int P_COL = 2 * KC;          // P: PMAX columns
constexpr uint64_t kLimitNs = 2000000000ull;
static_assert(P_COL + PMAX <= (int)TMEM_COLS, "TMEM budget");

struct Smem {
  uint8_t q[2][QBYTES];
  uint8_t k[NST][KBYTES];
  int32_t kidx[2][PMAX + TMAX];
  float2 xch[2][C][2][QR];
  uint8_t kreg[2][PMAX];
  uint64_t kfull[NST], kempty[NST], qfull[2], qempty[2], sfull[2], sempty[2], xbar[2], iready[2], idone[2], mdone;
  uint32_t tmem_base;
  int abort;
  uint32_t issued_k, issued_q;  // producer's final counters (for the drain after an abort)
};
}  // namespace s2f

int s2_fused_smem_bytes() { return (int)sizeof(s2f::Smem) + 1024; }
int s2_fused_threads() { return s2f::THREADS; }

namespace {

struct ItemGeom {
  int b, j0, M, n, img0, own_img, txt0, own_txt, nic, ntc, slot;
  int64_t rbase, t0;
};

__device__ __forceinline__ ItemGeom item_geom(const Stage2TcParams& p, int4 it, int rank) {
  using namespace s2f;
  ItemGeom g;
  g.b = it.x;
  g.j0 = it.y;
  g.slot = it.z;
  g.rbase = p.bt.row_off[g.b];
  g.t0 = p.bt.text_off[g.b];
  g.M = (int)(p.bt.text_off[g.b + 1] - g.t0);
  g.n = p.n1[g.b];
  const int per = (g.n + C - 1) / C;
  g.img0 = rank * per;
  g.own_img = max(0, min(per, g.n - g.img0));
  const int n_txt = p.has_text ? min(g.j0 + QR, g.M) : 0;
  const int per_t = (n_txt + C - 1) / C;
  g.txt0 = rank * per_t;
  g.own_txt = max(0, min(per_t, n_txt - g.txt0));
  g.nic = (g.own_img + KC - 1) / KC;
  g.ntc = (g.own_txt + KC - 1) / KC;
  return g;
}

__device__ __forceinline__ void fail(s2f::Smem& sm, int* status) {
  sm.abort = 1;
  set_status(status, OCCAM_ERR_TIMEOUT);
}

__device__ __forceinline__ float warp_max_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

}  // namespace

__global__ void __launch_bounds__(s2f::THREADS, 1)
    s2_fused_kernel(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapK,
                    const __grid_constant__ CUtensorMap mapKt, Stage2TcParams p) {
  using namespace s2f;
  extern __shared__ unsigned char smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rank = (int)tc::cluster_rank();
  const int nF = p.counters[CNT_NF];
  const int cid = (int)tc::cluster_id_x(), ncl = (int)tc::nclusters_x();
  volatile int* abort = &sm.abort;

  if (tid == 0) {
    for (int i = 0; i < NST; ++i) { tc::bar_init(&sm.kfull[i], NPROD * 32); tc::bar_init(&sm.kempty[i], 1); }
    for (int i = 0; i < 2; ++i) {
      tc::bar_init(&sm.qfull[i], 1);
      tc::bar_init(&sm.qempty[i], 1);
      tc::bar_init(&sm.sfull[i], 1);
      tc::bar_init(&sm.sempty[i], 4);
      tc::bar_init(&sm.xbar[i], NEPI * C);
      tc::bar_init(&sm.iready[i], NPROD * 32);
      tc::bar_init(&sm.idone[i], NEPI);
    }
    tc::bar_init(&sm.mdone, 1);
    sm.abort = 0;
    sm.issued_k = 0;
    sm.issued_q = 0;
    tc::bar_fence_init();
    tc::prefetch_map(&mapQ);
    tc::prefetch_map(&mapK);
    tc::prefetch_map(&mapKt);
  }
  if (warp == MMA_WARP) tc::tmem_alloc(&sm.tmem_base, TMEM_COLS);
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  // peers' barriers must be initialised before anyone arrives on them remotely
  tc::cluster_sync_all();
  const uint32_t tmem = sm.tmem_base;
  const int H = p.H;

  if (warp < NPROD) {
    // ------------------------------------------------------------ producers
    // 96 threads; piece q = pt + 96 i (q < 1024) of a chunk is 16 bytes of key
    // row (q >> 4), head slice bytes 16 * (q & 15); it lands at the row's
    // 128-byte line of its K-block with the 16-byte chunk index XOR (row & 7).
    const int pt = tid;
    uint32_t qcnt = 0, kcnt = 0;
    int ii = 0;
    const int64_t HD = (int64_t)H * 128;
    for (int item = cid; item < nF; item += ncl, ++ii) {
      const ItemGeom g = item_geom(p, p.items[item], rank);
      const int ib = ii & 1;
      if (*abort || !tc::bar_wait(&sm.idone[ib], ((ii >> 1) & 1) ^ 1, abort, kLimitNs)) { fail(sm, p.status); break; }
      for (int i = pt; i < g.own_img; i += NPROD * 32) {
        const int row = p.dense[g.rbase + g.img0 + i];
        sm.kidx[ib][i] = row;
        sm.kreg[ib][i] = p.role[row];
      }
      for (int i = pt; i < g.own_txt; i += NPROD * 32) sm.kidx[ib][PMAX + i] = (int)(g.t0 + g.txt0 + i);
      tc::bar_arrive(&sm.iready[ib]);
      if (!tc::bar_wait(&sm.iready[ib], (ii >> 1) & 1, abort, kLimitNs)) { fail(sm, p.status); break; }
      const int nch = 2 * g.nic + g.ntc;
      bool ok = true;
      for (int h = 0; h < H && ok; ++h) {
        if (pt == 0) {
          const int qb = qcnt & 1;
          if (!tc::bar_wait(&sm.qempty[qb], ((qcnt >> 1) & 1) ^ 1, abort, kLimitNs)) {
            fail(sm, p.status);
            ok = false;
          } else {
            tc::bar_expect_tx(&sm.qfull[qb], QBYTES);
            tc::tma_load_2d(sm.q[qb], &mapQ, h * 128, (int)(g.t0 + g.j0), &sm.qfull[qb]);
            tc::tma_load_2d(sm.q[qb] + QBYTES / 2, &mapQ, h * 128 + 64, (int)(g.t0 + g.j0), &sm.qfull[qb]);
          }
        }
        ++qcnt;
        for (int ci = 0; ci < nch && ok; ++ci) {
          const int st = kcnt % NST;
          if (!tc::bar_wait(&sm.kempty[st], ((kcnt / NST) & 1) ^ 1, abort, kLimitNs)) {
            fail(sm, p.status);
            ok = false;
            break;
          }
          const bool is_txt = (ci >= g.nic) && (ci < g.nic + g.ntc);
          const int c = ci < g.nic ? ci : (is_txt ? ci - g.nic : ci - g.nic - g.ntc);
          const int* rows = is_txt ? &sm.kidx[ib][PMAX + c * KC] : &sm.kidx[ib][c * KC];
          const int nv = is_txt ? min(KC, g.own_txt - c * KC) : min(KC, g.own_img - c * KC);
          const __nv_bfloat16* base = is_txt ? p.Kt : p.K;
          uint8_t* dst = sm.k[st];
#pragma unroll
          for (int i = 0; i < (KC * 16 + NPROD * 32 - 1) / (NPROD * 32); ++i) {
            const int q = pt + NPROD * 32 * i;
            if (q >= KC * 16) break;
            const int key = q >> 4, c16 = q & 15;
            const int kb = c16 >> 3, cc = c16 & 7;
            const bool v = key < nv;
            const __nv_bfloat16* src = base + (v ? (int64_t)rows[key] * HD + h * 128 + c16 * 8 : 0);
            tc::cp_async16(dst + kb * (KBYTES / 2) + key * 128 + ((cc ^ (key & 7)) << 4), src, v ? 16 : 0);
          }
          tc::cp_async_arrive(&sm.kfull[st]);
          ++kcnt;
        }
      }
      if (!ok) break;
    }
    if (pt == 0) {
      sm.issued_k = kcnt;
      sm.issued_q = qcnt;
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
  } else if (warp == MMA_WARP) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      uint32_t qcnt = 0, kcnt = 0, scnt = 0;
      for (int item = cid; item < nF && !*abort; item += ncl) {
        const ItemGeom g = item_geom(p, p.items[item], rank);
        const int nch = 2 * g.nic + g.ntc;
        for (int h = 0; h < H && !*abort; ++h) {
          const int qb = qcnt & 1;
          if (!tc::bar_wait(&sm.qfull[qb], (qcnt >> 1) & 1, abort, kLimitNs)) { fail(sm, p.status); break; }
          for (int ci = 0; ci < nch; ++ci) {
            const int st = kcnt % NST;
            const int sb = scnt & 1;
            if (!tc::bar_wait(&sm.kfull[st], (kcnt / NST) & 1, abort, kLimitNs) ||
                !tc::bar_wait(&sm.sempty[sb], ((scnt >> 1) & 1) ^ 1, abort, kLimitNs)) {
              fail(sm, p.status);
              break;
            }
            tc::fence_proxy_async();
            tc::fence_after();
            const uint32_t d = tmem + S_COL + sb * KC;
            const uint32_t qa = tc::su32(sm.q[qb]), kbase = tc::su32(sm.k[st]);
#pragma unroll
            for (int k = 0; k < 8; ++k) {
              const int kb = k >> 2, kk = k & 3;
              tc::mma_bf16(d, tc::sdesc_sw128(qa + kb * (QBYTES / 2) + kk * 32),
                           tc::sdesc_sw128(kbase + kb * (KBYTES / 2) + kk * 32), IDESC, k > 0 ? 1u : 0u);
            }
            tc::mma_commit(&sm.sfull[sb]);
            tc::mma_commit(&sm.kempty[st]);
            ++kcnt;
            ++scnt;
          }
          tc::mma_commit(&sm.qempty[qb]);
          ++qcnt;
        }
      }
      // every MMA issued by this thread has completed once this barrier flips
      tc::mma_commit(&sm.mdone);
      if (!tc::bar_wait(&sm.mdone, 0, nullptr, kLimitNs)) set_status(p.status, OCCAM_ERR_TIMEOUT);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------ epilogue
    const int ew = warp - EPI_WARP0;    // 0..NEPI-1
    const int half = ew >> 2;           // which chunks (index parity) this warp takes
    const int quad = warp & 3;          // TMEM lane quadrant this warp may access
    const int j = quad * 32 + lane;     // text row of this thread inside the tile
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    const float sl2 = p.scale_log2;
    const float invH = 1.0f / (float)H;
    const uint32_t sbuf = tmem + lane_base + S_COL + half * KC;
    uint32_t scnt = 0, xcnt = 0;
    int ii = 0;
    for (int item = cid; item < nF; item += ncl, ++ii) {
      const ItemGeom g = item_geom(p, p.items[item], rank);
      const int ib = ii & 1;
      if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.iready[ib], (ii >> 1) & 1, nullptr, kLimitNs))) { fail(sm, p.status); break; }
      const bool vrow = g.j0 + j < g.M;
      const bool wvalid = __any_sync(0xffffffffu, vrow);  // warp-uniform: any real text row here
      const int jj = g.j0 + j;
      bool ok = true;
      uint32_t pstart = 0;  // chunk counter at the start of the last P pass
      for (int h = 0; h < H && ok; ++h) {
        // ---- statistics over this warp's chunks of the CTA's keys
        float m = -INFINITY, z = 0.f;
        for (int ci = 0; ci < g.nic + g.ntc; ++ci, ++scnt) {
          if ((int)(scnt & 1) != half) continue;
          if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.sfull[half], (scnt >> 1) & 1, nullptr, kLimitNs))) { ok = false; break; }
          const bool is_txt = ci >= g.nic;
          const int c = is_txt ? ci - g.nic : ci;
          const int nv = is_txt ? min(KC, g.own_txt - c * KC) : min(KC, g.own_img - c * KC);
          const int tbase = g.txt0 + c * KC;  // sample-relative text index of column 0
          const int lim = vrow ? (is_txt ? min(nv, jj - tbase + 1) : nv) : 0;
#pragma unroll
          for (int hf = 0; hf < 2; ++hf) {
            uint32_t v[32];
            if (wvalid) {
              tc::fence_after();
              tc::tmem_ld32(sbuf + hf * 32, v);
              tc::tmem_wait_ld();
            }
            if (hf == 1) {
              tc::fence_before();
              __syncwarp();
              if (lane == 0) tc::bar_arrive(&sm.sempty[half]);
            }
            const int l2 = lim - hf * 32;  // valid columns in this half
            if (l2 > 0) {
              float cm0 = -INFINITY, cm1 = -INFINITY;
#pragma unroll
              for (int col = 0; col < 32; col += 2) {
                if (col < l2) cm0 = fmaxf(cm0, __uint_as_float(v[col]));
                if (col + 1 < l2) cm1 = fmaxf(cm1, __uint_as_float(v[col + 1]));
              }
              const float mn = fmaxf(m, fmaxf(cm0, cm1) * sl2);
              float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
#pragma unroll
              for (int col = 0; col < 32; col += 4) {
                if (col < l2) a0 += tc::ex2(fmaf(__uint_as_float(v[col]), sl2, -mn));
                if (col + 1 < l2) a1 += tc::ex2(fmaf(__uint_as_float(v[col + 1]), sl2, -mn));
                if (col + 2 < l2) a2 += tc::ex2(fmaf(__uint_as_float(v[col + 2]), sl2, -mn));
                if (col + 3 < l2) a3 += tc::ex2(fmaf(__uint_as_float(v[col + 3]), sl2, -mn));
              }
              z = (m == -INFINITY ? 0.f : z * tc::ex2(m - mn)) + ((a0 + a1) + (a2 + a3));
              m = mn;
            }
          }
        }
        if (!ok) break;
        // ---- exchange (max, sum) with every epilogue warp of the cluster
        const int slot = xcnt & 1;
        for (int r = 0; r < C; ++r) tc::st_cluster_f2(&sm.xch[slot][rank][half][j], (uint32_t)r, m, z);
        __syncwarp();
        if (lane == 0)
          for (int r = 0; r < C; ++r) tc::bar_arrive_remote(&sm.xbar[slot], (uint32_t)r);
        if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.xbar[slot], (xcnt >> 1) & 1, nullptr, kLimitNs, true))) { ok = false; break; }
        ++xcnt;
        float Mx = -INFINITY;
#pragma unroll
        for (int r = 0; r < C; ++r)
          Mx = fmaxf(Mx, fmaxf(sm.xch[slot][r][0][j].x, sm.xch[slot][r][1][j].x));
        float Z = 0.f;
#pragma unroll
        for (int r = 0; r < C; ++r)
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            const float2 e = sm.xch[slot][r][hh][j];
            if (e.y > 0.f) Z += e.y * tc::ex2(e.x - Mx);
          }
        const float f = (Z > 0.f) ? 1.0f / Z : 0.f;
        // ---- probabilities of the CTA's S1 keys, summed over heads in TMEM
        pstart = scnt;
        for (int c = 0; c < g.nic; ++c, ++scnt) {
          if ((int)(scnt & 1) != half) continue;
          if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.sfull[half], (scnt >> 1) & 1, nullptr, kLimitNs))) { ok = false; break; }
          const uint32_t pa = tmem + lane_base + P_COL + c * KC;
          const int nv = min(KC, g.own_img - c * KC);
          const float mf = vrow ? Mx : INFINITY;   // rows past M contribute 0
          // two halves of 32 columns keep the live registers down
#pragma unroll
          for (int hf = 0; hf < 2; ++hf) {
            uint32_t v[32], w[32];
            if (wvalid) {
              tc::fence_after();
              tc::tmem_ld32(sbuf + hf * 32, v);
              if (h > 0) tc::tmem_ld32(pa + hf * 32, w);
              tc::tmem_wait_ld();
            }
            if (hf == 1) {  // the S buffer is free once both halves are in registers
              tc::fence_before();
              __syncwarp();
              if (lane == 0) tc::bar_arrive(&sm.sempty[half]);
            }
            if (wvalid) {
#pragma unroll
              for (int col = 0; col < 32; ++col) {
                const float pv = (hf * 32 + col < nv) ? tc::ex2(fmaf(__uint_as_float(v[col]), sl2, -mf)) * f : 0.f;
                w[col] = __float_as_uint(h > 0 ? __uint_as_float(w[col]) + pv : pv);
              }
              tc::tmem_st32(pa + hf * 32, w);
            }
          }
        }
        if (wvalid) tc::tmem_wait_st();
        // order this warp's P stores before the next head's exchange arrival
        tc::fence_before();
      }
      if (!ok) { fail(sm, p.status); break; }
      // ---- column reductions of P over this warp's 32 rows, for the chunks
      // this warp wrote in the last head (so no other warp's stores are
      // involved): column max -> s2 (atomicMax), register columns -> this
      // warp's partial of s2(r)
      float regacc = 0.f;
      if (wvalid) {
        tc::fence_after();
        for (int c = (int)((pstart + half) & 1); c < g.nic; c += 2) {
          const int nv = min(KC, g.own_img - c * KC);
          for (int hf = 0; hf < 2; ++hf) {
            uint32_t w[32];
            tc::tmem_ld32(tmem + lane_base + P_COL + c * KC + hf * 32, w);
            tc::tmem_wait_ld();
#pragma unroll
            for (int col = 0; col < 32; ++col) {
              const float x = vrow ? __uint_as_float(w[col]) : 0.f;
              const float mx = warp_max_f(x);
              const float su = warp_sum_f(x);
              if (lane == 0 && hf * 32 + col < nv) {
                const int key = c * KC + hf * 32 + col;
                if (sm.kreg[ib][key]) regacc += su * invH;
                else atomicMax(reinterpret_cast<int*>(&p.s2[sm.kidx[ib][key]]), __float_as_int(mx * invH));
              }
            }
          }
        }
      }
      if (lane == 0) {
        p.refpart[g.slot + rank * NEPI + ew] = regacc;
        __threadfence();
        const int nslots = p.slot_off[g.b + 1] - p.slot_off[g.b];
        if (atomicAdd(&p.done[g.b], 1) == nslots - 1) {
          __threadfence();
          float acc = 0.f;
          for (int i = p.slot_off[g.b]; i < p.slot_off[g.b + 1]; ++i) acc += *((volatile float*)&p.refpart[i]);
          const int R = p.bt.reg_off[p.bt.seg_first[g.b + 1]] - p.bt.reg_off[p.bt.seg_first[g.b]];
          const float r2 = (R > 0 && g.M > 0) ? acc / ((float)R * (float)g.M) : 0.f;
          p.ref2[g.b] = r2;
          p.tau2[g.b] = p.lambda2 * r2;
        }
      }
      __syncwarp();
      if (lane == 0) tc::bar_arrive(&sm.idone[ib]);
    }
  }

  // ------------------------------------------------------------ teardown
  tc::fence_before();
  __syncthreads();
  if (sm.abort && tid == 0) {
    // drain the last query-tile copies (TMA) issued into each buffer; the
    // producers' cp.async copies were drained by cp.async.wait_all
    const uint32_t q1 = sm.issued_q;
    for (uint32_t i = (q1 > 2 ? q1 - 2 : 0); i < q1; ++i)
      tc::bar_wait(&sm.qfull[i & 1], (i >> 1) & 1, nullptr, kLimitNs / 8);
  }
  __syncthreads();
  tc::fence_after();
  if (warp == MMA_WARP) tc::tmem_dealloc(tmem, TMEM_COLS);
  // peers may still write into this CTA's exchange buffers until here
  tc::cluster_sync_all();
}

}  // namespace occam
