// stage2_tc.cu -- fused Stage-II scoring on the 5th-generation tensor cores
// (tcgen05 + TMEM), for samples whose S1 fits a 4-CTA cluster.
//
// What it computes (Sec. 3.5, Eq. 7; App. A, Eqs. 15-16): for sample b, text
// token j and head h, A_{j,h} = softmax over {S1 rows of b} u {text keys 0..j}
// of q_{j,h} k^T / sqrt(d2); P[j, v] = sum_h A_{j,h}(v); s2(v) = max_j P[j, v] / H
// for visual S1 rows and the registers' sum_j P[j, r] / H for s2(r).
//
// Work item = (sample, tile of 128 text rows), processed by one cluster of C
// CTAs (C = 4, or 8 for samples with more S1 keys). The text rows are the 128
// TMEM lanes; each CTA owns 1/C of the sample's S1 keys and of the causal
// text keys. Per head:
//   1. three producer warps stream the CTA's key rows in 64-key chunks with
//      16-byte cp.async into the 128-byte-swizzled operand layout (S1 rows
//      are gathered by index straight from K2: pruned rows are never read,
//      every key row is read once per text tile); the head's 128 x 128 query
//      tile arrives by TMA;
//   2. one thread issues S = Q K^T per chunk (tcgen05.mma, bf16 in, fp32 in
//      TMEM): text-key chunks into a two-deep scratch ring, S1-key chunks
//      into a per-head TMEM buffer E (two buffers, alternating by head);
//   3. eight epilogue warps (two per TMEM lane quadrant, one thread per text
//      row) each own one 32-column half of every chunk. A warp turns its
//      logits into exp2(l - cmax) (cmax: the row max of that half-chunk, kept
//      in a register), writes them back over S1-key logits in E, and keeps
//      the row's running softmax max / sum;
//   4. the (max, sum) pairs go to every epilogue warp of the cluster with
//      asynchronous distributed-shared-memory stores that complete on an
//      mbarrier of the receiving CTA (no fences). The exchange of head h is
//      awaited only after head h+1's statistics, so its latency is hidden;
//   5. then every warp adds exp2(cmax - max) / sum * E over its own columns to
//      the head-summed probabilities P, which live in registers for the
//      whole item.
// After the last head every warp reduces its P columns over its 32 rows:
// column max -> s2 (atomicMax on the fp32 bit pattern, exact and order-free
// since P >= 0), register columns -> a partial of s2(r) reduced in fixed order.
#include "common.cuh"
#include "kernels.cuh"
#include "tc5.cuh"

namespace occam {

namespace s2f {
constexpr int QR = 128;                // text rows per item (TMEM lanes)
constexpr int KC = 64;                 // keys per chunk (MMA N)
constexpr int NST = 4;                 // key-chunk ring stages
constexpr int PMAX = kFusedMaxOwnImg;  // max S1 keys per CTA
constexpr int NIC_MAX = PMAX / KC;     // S1-key chunks per CTA
constexpr int TMAX = kFusedMaxOwnTxt;  // max text keys per CTA
constexpr int QBYTES = QR * 256;       // one head's query tile: 2 K-blocks x 128 rows x 128 B
constexpr int KBYTES = KC * 256;       // one chunk: 2 K-blocks x 64 rows x 128 B
constexpr int NPROD = 3;               // producer warps (0-2); warp 3 issues MMAs; then the epilogue warps
constexpr int MMA_WARP = NPROD;
constexpr int EPI_WARP0 = NPROD + 1;
constexpr int NEPI = kFusedEpiWarps;   // two per TMEM lane quadrant
constexpr int THREADS = (NPROD + 1 + NEPI) * 32;
constexpr int NXS = 4;                 // exchange slots (the exchange runs one head behind)
// register split: warpgroup 0 (producers + MMA issuer) shrinks to REG_LOW per
// thread, the two epilogue warpgroups grow to REG_HIGH; the sum must stay
// within what the CTA was launched with (checked on the host before launch)
constexpr int REG_LOW = 88, REG_HIGH = 208;
constexpr int REG_NEEDED = 128 * REG_LOW + (THREADS - 128) * REG_HIGH;
static_assert(NPROD + 1 == 4 && (THREADS - 128) % 128 == 0, "warpgroup 0 = producers + MMA warp");
constexpr uint32_t IDESC = tc::idesc_bf16(128, KC);
constexpr uint32_t TMEM_COLS = 512;
constexpr int S_COL = 0;               // two scratch buffers (text-key chunks), KC columns each
constexpr int E_COL = 2 * KC;          // two E buffers (by head parity), PMAX columns each
static_assert(E_COL + 2 * PMAX <= (int)TMEM_COLS, "TMEM budget");
static_assert(PMAX % KC == 0, "E buffers hold whole chunks");
constexpr uint64_t kLimitNs = 2000000000ull;

template <int C>
struct Smem {
  static constexpr uint32_t XBYTES = C * NEPI * 32 * 8;  // exchange bytes one CTA receives per head
  uint8_t q[2][QBYTES];
  uint8_t k[NST][KBYTES];
  int32_t kidx[2][PMAX + TMAX];
  float2 xch[NXS][C][2][QR];          // (max, sum) per (slot, CTA, epilogue half, row)
  uint8_t kreg[2][PMAX];
  uint64_t kfull[NST], kempty[NST], qfull[2], qempty[2], sfull[2], sempty[2], efull[2][NIC_MAX], efree[2],
      xbar[NXS], iready[2], idone[2], mdone;
  uint32_t tmem_base;
  int abort;
  uint32_t issued_q;
};
}  // namespace s2f

int s2_fused_smem_bytes(int C) {
  return (int)(C == 8 ? sizeof(s2f::Smem<8>) : sizeof(s2f::Smem<4>)) + 1024;
}
int s2_fused_threads() { return s2f::THREADS; }

namespace {

struct ItemGeom {
  int b, j0, M, n, img0, own_img, txt0, own_txt, nic, ntc, slot;
  int64_t rbase, t0;
};

template <int C>
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

template <class SM>
__device__ __forceinline__ void fail(SM& sm, int* status) {
  sm.abort = 1;
  set_status(status, OCCAM_ERR_TIMEOUT);
}

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Statistics of one thread's row over a 32-column half-chunk of logits at
// TMEM address sa (warp-collective): cm = max of the first `lim` columns in
// log2 units (-inf if none), a = sum over them of exp2(l * sl2 - cm). With
// STORE the exponentials (0 past lim) are written back over the logits; the
// caller waits for that store before the values are read again.
template <bool STORE>
__device__ __forceinline__ void half_stats(uint32_t sa, int lim, float sl2, float& cm, float& a) {
  cm = -INFINITY;
  a = 0.f;
  if (__all_sync(0xffffffffu, lim <= 0)) return;
  const bool full = __all_sync(0xffffffffu, lim >= 32);
  uint32_t v[32];
  tc::fence_after();
  tc::tmem_ld32(sa, v);
  tc::tmem_wait_ld();
  if (full) {
    float t[11];
#pragma unroll
    for (int i = 0; i < 10; ++i)
      t[i] = tc::fmax3(__uint_as_float(v[3 * i]), __uint_as_float(v[3 * i + 1]), __uint_as_float(v[3 * i + 2]));
    t[10] = fmaxf(__uint_as_float(v[30]), __uint_as_float(v[31]));
    const float mx = fmaxf(tc::fmax3(tc::fmax3(t[0], t[1], t[2]), tc::fmax3(t[3], t[4], t[5]), tc::fmax3(t[6], t[7], t[8])),
                           fmaxf(t[9], t[10]));
    cm = mx * sl2;
    const float2 sc = make_float2(sl2, sl2), off = make_float2(-cm, -cm);
    float2 acc0 = make_float2(0.f, 0.f), acc1 = acc0;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      float2 x = __ffma2_rn(make_float2(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1])), sc, off);
      x.x = tc::ex2(x.x);
      x.y = tc::ex2(x.y);
      if (i & 1) acc1 = __fadd2_rn(acc1, x);
      else acc0 = __fadd2_rn(acc0, x);
      v[2 * i] = __float_as_uint(x.x);
      v[2 * i + 1] = __float_as_uint(x.y);
    }
    a = (acc0.x + acc0.y) + (acc1.x + acc1.y);
  } else {
    float c0 = -INFINITY, c1 = -INFINITY;
#pragma unroll
    for (int col = 0; col < 32; col += 2) {
      if (col < lim) c0 = fmaxf(c0, __uint_as_float(v[col]));
      if (col + 1 < lim) c1 = fmaxf(c1, __uint_as_float(v[col + 1]));
    }
    cm = fmaxf(c0, c1) * sl2;
    float a0 = 0.f, a1 = 0.f;
#pragma unroll
    for (int col = 0; col < 32; col += 2) {
      const float e0 = (col < lim) ? tc::ex2(fmaf(__uint_as_float(v[col]), sl2, -cm)) : 0.f;
      const float e1 = (col + 1 < lim) ? tc::ex2(fmaf(__uint_as_float(v[col + 1]), sl2, -cm)) : 0.f;
      a0 += e0;
      a1 += e1;
      v[col] = __float_as_uint(e0);
      v[col + 1] = __float_as_uint(e1);
    }
    a = a0 + a1;
  }
  if (STORE) tc::tmem_st32(sa, v);
}

// merges a half-chunk's (cm, a) into the row's running softmax (m, z), log2 units
__device__ __forceinline__ void online_merge(float& m, float& z, float cm, float a) {
  if (cm != -INFINITY) {
    const float mn = fmaxf(m, cm);
    z = (m == -INFINITY ? 0.f : z * tc::ex2(m - mn)) + a * tc::ex2(cm - mn);
    m = mn;
  }
}

}  // namespace

template <int C>
__global__ void __launch_bounds__(s2f::THREADS, 1)
    s2_fused_kernel(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapK,
                    const __grid_constant__ CUtensorMap mapKt, Stage2TcParams p) {
  using namespace s2f;
  extern __shared__ unsigned char smem_raw[];
  Smem<C>& sm = *reinterpret_cast<Smem<C>*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rank = (int)tc::cluster_rank();
  const int nF = p.counters[C == 8 ? CNT_NF8 : CNT_NF];
  const int cid = (int)tc::cluster_id_x(), ncl = (int)tc::nclusters_x();
  volatile int* abort = &sm.abort;
  (void)mapK;
  (void)mapKt;

  if (tid == 0) {
    for (int i = 0; i < NST; ++i) { tc::bar_init(&sm.kfull[i], NPROD * 32); tc::bar_init(&sm.kempty[i], 1); }
    for (int i = 0; i < 2; ++i) {
      tc::bar_init(&sm.qfull[i], 1);
      tc::bar_init(&sm.qempty[i], 1);
      tc::bar_init(&sm.sfull[i], 1);
      tc::bar_init(&sm.sempty[i], NEPI);
      for (int c = 0; c < NIC_MAX; ++c) tc::bar_init(&sm.efull[i][c], 1);
      tc::bar_init(&sm.efree[i], NEPI);
      tc::bar_init(&sm.iready[i], NPROD * 32);
      tc::bar_init(&sm.idone[i], NEPI);
    }
    // one local arrival (with the expected byte count) plus the peers'
    // asynchronous stores complete each phase of an exchange slot
    for (int i = 0; i < NXS; ++i) tc::bar_init(&sm.xbar[i], 1);
    tc::bar_init(&sm.mdone, 1);
    sm.abort = 0;
    sm.issued_q = 0;
    tc::bar_fence_init();
    for (int i = 0; i < NXS; ++i) tc::bar_expect_tx(&sm.xbar[i], Smem<C>::XBYTES);
    tc::prefetch_map(&mapQ);
  }
  if (warp == MMA_WARP) tc::tmem_alloc(&sm.tmem_base, TMEM_COLS);
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  // peers' barriers must be initialised before anyone arrives on them remotely
  tc::cluster_sync_all();
  const uint32_t tmem = sm.tmem_base;
  const int H = p.H;

  if (warp < 4) {
    // warpgroup 0: producers and the MMA issuer give registers back
    tc::setmaxnreg_dec<REG_LOW>();
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
        const ItemGeom g = item_geom<C>(p, p.items[item], rank);
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
        const int nch = g.nic + g.ntc;
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
            const bool is_txt = ci < g.ntc;  // text chunks first: they do not wait for an E buffer
            const int c = is_txt ? ci : ci - g.ntc;
            const int* rows = is_txt ? &sm.kidx[ib][PMAX + c * KC] : &sm.kidx[ib][c * KC];
            const int nv = is_txt ? min(KC, g.own_txt - c * KC) : min(KC, g.own_img - c * KC);
            const __nv_bfloat16* base = is_txt ? p.Kt : p.K;
            uint8_t* dst = sm.k[st];
  #pragma unroll
            for (int i = 0; i < (KC * 16 + NPROD * 32 - 1) / (NPROD * 32); ++i) {
              const int q = pt + NPROD * 32 * i;
              if (q < KC * 16) {
                const int key = q >> 4, c16 = q & 15;
                const int kb = c16 >> 3, cc = c16 & 7;
                const bool v = key < nv;
                const __nv_bfloat16* src = base + (v ? (int64_t)rows[key] * HD + h * 128 + c16 * 8 : 0);
                tc::cp_async16(dst + kb * (KBYTES / 2) + key * 128 + ((cc ^ (key & 7)) << 4), src, v ? 16 : 0);
              }
            }
            tc::cp_async_arrive(&sm.kfull[st]);
            ++kcnt;
          }
        }
        if (!ok) break;
      }
      if (pt == 0) sm.issued_q = qcnt;
      asm volatile("cp.async.wait_all;" ::: "memory");
    } else {
      // ------------------------------------------------------------ MMA issuer
      if (lane == 0) {
        uint32_t qcnt = 0, kcnt = 0, tcnt = 0, hk = 0;
        for (int item = cid; item < nF && !*abort; item += ncl) {
          const ItemGeom g = item_geom<C>(p, p.items[item], rank);
          const int nch = g.nic + g.ntc;
          for (int h = 0; h < H && !*abort; ++h, ++hk) {
            const int qb = qcnt & 1;
            if (!tc::bar_wait(&sm.qfull[qb], (qcnt >> 1) & 1, abort, kLimitNs)) { fail(sm, p.status); break; }
            const int eb = hk & 1;
            bool ok = true;
            for (int ci = 0; ci < nch && ok; ++ci) {
              const bool is_txt = ci < g.ntc;
              const int st = kcnt % NST;
              uint32_t d;
              if (is_txt) {
                const int sb = tcnt & 1;
                ok = tc::bar_wait(&sm.sempty[sb], ((tcnt >> 1) & 1) ^ 1, abort, kLimitNs);
                d = tmem + S_COL + sb * KC;
              } else {
                // E[eb] is free once the probabilities of head hk - 2 were read out of it
                if (ci == g.ntc && hk >= 2) ok = tc::bar_wait(&sm.efree[eb], ((hk - 2) >> 1) & 1, abort, kLimitNs);
                d = tmem + E_COL + eb * PMAX + (ci - g.ntc) * KC;
              }
              if (ok) ok = tc::bar_wait(&sm.kfull[st], (kcnt / NST) & 1, abort, kLimitNs);
              if (!ok) {
                fail(sm, p.status);
                break;
              }
              tc::fence_proxy_async();
              tc::fence_after();
              const uint32_t qa = tc::su32(sm.q[qb]), kbase = tc::su32(sm.k[st]);
  #pragma unroll
              for (int k = 0; k < 8; ++k) {
                const int kb = k >> 2, kk = k & 3;
                tc::mma_bf16(d, tc::sdesc_sw128(qa + kb * (QBYTES / 2) + kk * 32),
                             tc::sdesc_sw128(kbase + kb * (KBYTES / 2) + kk * 32), IDESC, k > 0 ? 1u : 0u);
              }
              if (is_txt) {
                tc::mma_commit(&sm.sfull[tcnt & 1]);
                ++tcnt;
              } else {
                tc::mma_commit(&sm.efull[eb][ci - g.ntc]);
              }
              tc::mma_commit(&sm.kempty[st]);
              ++kcnt;
            }
            if (!ok) break;
            // the E-chunk barriers of chunks this item does not use still
            // complete once per head, so every barrier's phase follows the head index
            for (int c = g.nic; c < NIC_MAX; ++c) tc::mma_commit(&sm.efull[eb][c]);
            tc::mma_commit(&sm.qempty[qb]);
            ++qcnt;
          }
        }
        // every MMA issued by this thread has completed once this barrier flips
        tc::mma_commit(&sm.mdone);
        if (!tc::bar_wait(&sm.mdone, 0, nullptr, kLimitNs)) set_status(p.status, OCCAM_ERR_TIMEOUT);
      }
      __syncwarp();
    }
  } else {
    // warpgroups 1 and 2: the epilogue takes them
    tc::setmaxnreg_inc<REG_HIGH>();
    // ------------------------------------------------------------ epilogue
    const int ew = warp - EPI_WARP0;    // 0..NEPI-1
    const int half = ew >> 2;           // the 32-column half of every chunk this warp owns
    const int quad = warp & 3;          // TMEM lane quadrant this warp may access
    const int j = quad * 32 + lane;     // text row of this thread inside the tile
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    const float sl2 = p.scale_log2;
    const float invH = 1.0f / (float)H;
    const bool armer = ew == 0 && lane == 0;  // re-arms the exchange slots of this CTA
    uint32_t tcnt = 0, hk = 0;
    int ii = 0;
    for (int item = cid; item < nF; item += ncl, ++ii) {
      const ItemGeom g = item_geom<C>(p, p.items[item], rank);
      const int ib = ii & 1;
      if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.iready[ib], (ii >> 1) & 1, nullptr, kLimitNs))) { fail(sm, p.status); break; }
      const bool vrow = g.j0 + j < g.M;
      const bool wvalid = __any_sync(0xffffffffu, vrow);  // warp-uniform: any real text row here
      const int jj = g.j0 + j;
      float P[NIC_MAX][32];
#pragma unroll
      for (int c = 0; c < NIC_MAX; ++c)
#pragma unroll
        for (int b2 = 0; b2 < 32; ++b2) P[c][b2] = 0.f;
      float cmx[NIC_MAX];  // half-chunk maxima of the last head whose statistics were taken
#pragma unroll
      for (int c = 0; c < NIC_MAX; ++c) cmx[c] = -INFINITY;
      bool ok = true;
      // Step s takes the text-key statistics of head s, then adds head s-1
      // into P (which frees head s-1's E buffer for head s+1's MMAs while
      // this step still works on head s), then the S1-key statistics of head
      // s, and finally posts head s's (max, sum).
      for (int step = 0; step <= H && ok; ++step) {
        const uint32_t hcur = hk + step;  // global index of head `step` of this item
        float m = -INFINITY, z = 0.f;
        if (step < H) {
          // ---- text-key chunks of head `step` (scratch ring)
          for (int c = 0; c < g.ntc; ++c, ++tcnt) {
            const int sb = tcnt & 1;
            if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.sfull[sb], (tcnt >> 1) & 1, nullptr, kLimitNs))) { ok = false; break; }
            if (wvalid) {
              const int nv = min(KC, g.own_txt - c * KC);
              const int tbase = g.txt0 + c * KC + half * 32;  // sample-relative text index of this half's column 0
              const int lim = vrow ? min(nv - half * 32, jj - tbase + 1) : 0;
              float cm, a;
              half_stats<false>(tmem + lane_base + S_COL + sb * KC + half * 32, lim, sl2, cm, a);
              online_merge(m, z, cm, a);
            }
            tc::fence_before();
            __syncwarp();
            if (lane == 0) tc::bar_arrive(&sm.sempty[sb]);
          }
        }
        if (ok && step >= 1) {
          // ---- probabilities of head step-1 over this warp's columns, added into P
          const uint32_t hp = hcur - 1;
          const int slot = hp & (NXS - 1);
          const int eb = hp & 1;
          if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.xbar[slot], (hp / NXS) & 1, nullptr, kLimitNs, true))) {
            ok = false;
          } else {
            if (wvalid) {
              float Mx = -INFINITY;
#pragma unroll
              for (int r = 0; r < C; ++r) Mx = tc::fmax3(Mx, sm.xch[slot][r][0][j].x, sm.xch[slot][r][1][j].x);
              float Z = 0.f;
#pragma unroll
              for (int r = 0; r < C; ++r)
#pragma unroll
                for (int hh = 0; hh < 2; ++hh) {
                  const float2 e = sm.xch[slot][r][hh][j];
                  if (e.y > 0.f) Z += e.y * tc::ex2(e.x - Mx);
                }
              const float invZ = (vrow && Z > 0.f) ? 1.0f / Z : 0.f;
              tc::fence_after();
#pragma unroll
              for (int c = 0; c < NIC_MAX; ++c) {
                if (c < g.nic) {
                  const float f = (invZ > 0.f && cmx[c] != -INFINITY) ? tc::ex2(cmx[c] - Mx) * invZ : 0.f;
                  uint32_t v[32];
                  tc::tmem_ld32(tmem + lane_base + E_COL + eb * PMAX + c * KC + half * 32, v);
                  tc::tmem_wait_ld();
                  const float2 ff = make_float2(f, f);
#pragma unroll
                  for (int i = 0; i < 16; ++i) {
                    const float2 r2 = __ffma2_rn(make_float2(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1])),
                                                 ff, make_float2(P[c][2 * i], P[c][2 * i + 1]));
                    P[c][2 * i] = r2.x;
                    P[c][2 * i + 1] = r2.y;
                  }
                }
              }
            }
            tc::fence_before();
            __syncwarp();
            if (lane == 0) tc::bar_arrive(&sm.efree[eb]);
            // the slot's phase for head hp is complete: arm it for head hp + NXS
            if (armer) tc::bar_expect_tx(&sm.xbar[slot], Smem<C>::XBYTES);
          }
        }
        if (ok && step < H) {
          // ---- S1-key chunks of head `step` (E buffer), then the exchange
          const int eb = hcur & 1;
#pragma unroll
          for (int c = 0; c < NIC_MAX; ++c) {
            cmx[c] = -INFINITY;
            if (ok && c < g.nic) {
              if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.efull[eb][c], (hcur >> 1) & 1, nullptr, kLimitNs))) {
                ok = false;
              } else if (wvalid) {
                const int lim = vrow ? min(KC, g.own_img - c * KC) - half * 32 : 0;
                float a;
                half_stats<true>(tmem + lane_base + E_COL + eb * PMAX + c * KC + half * 32, lim, sl2, cmx[c], a);
                online_merge(m, z, cmx[c], a);
              }
            }
          }
          if (wvalid) tc::tmem_wait_st();
          tc::fence_before();
          if (ok) {
            // ---- post this head's (max, sum) to every epilogue warp of the cluster
            const int slot = hcur & (NXS - 1);
#pragma unroll
            for (int r = 0; r < C; ++r)
              tc::st_async_f2(&sm.xch[slot][rank][half][j], &sm.xbar[slot], (uint32_t)r, m, z);
          }
        }
      }
      hk += H;
      if (!ok) { fail(sm, p.status); break; }
      // ---- column reductions of P over this warp's 32 rows: column max ->
      // s2 (atomicMax), register columns -> this warp's partial of s2(r)
      float regacc = 0.f;
      if (wvalid) {
#pragma unroll
        for (int c = 0; c < NIC_MAX; ++c) {
          if (c < g.nic) {
            // transpose-reduce over the 32 rows of this warp: afterwards lane l
            // holds the max (and, where a register key is among the columns,
            // the sum) of this warp's column l of chunk c -- 31 shuffles each
            const int key = c * KC + half * 32 + lane;
            const bool live = key < g.own_img;
            const bool is_reg = live && sm.kreg[ib][key];
            float t[32];
#pragma unroll
            for (int col = 0; col < 32; ++col) t[col] = vrow ? P[c][col] : 0.f;
#pragma unroll
            for (int sft = 16; sft >= 1; sft >>= 1) {
              const bool up = (lane & sft) != 0;
#pragma unroll
              for (int i = 0; i < sft; ++i) {
                const float send = up ? t[i] : t[i + sft];
                const float keep = up ? t[i + sft] : t[i];
                t[i] = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, sft));
              }
            }
            if (live && !is_reg) atomicMax(reinterpret_cast<int*>(&p.s2[sm.kidx[ib][key]]), __float_as_int(t[0] * invH));
            float rc = 0.f;
            if (__any_sync(0xffffffffu, is_reg)) {
#pragma unroll
              for (int col = 0; col < 32; ++col) t[col] = vrow ? P[c][col] : 0.f;
#pragma unroll
              for (int sft = 16; sft >= 1; sft >>= 1) {
                const bool up = (lane & sft) != 0;
#pragma unroll
                for (int i = 0; i < sft; ++i) {
                  const float send = up ? t[i] : t[i + sft];
                  const float keep = up ? t[i + sft] : t[i];
                  t[i] = keep + __shfl_xor_sync(0xffffffffu, send, sft);
                }
              }
              if (is_reg) rc = t[0] * invH;
            }
            regacc += warp_sum_f(rc);
          }
        }
      }
      if (lane == 0) {
        p.refpart[g.slot + rank * NEPI + ew] = regacc;  // C * NEPI slots per item
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
  if (sm.abort && tid == 0) {
    // after an abort, peers' asynchronous exchange stores may still be in
    // flight towards this CTA: give them time to land before it can exit
    const uint64_t t0 = tc::globaltimer();
    while (tc::globaltimer() - t0 < 100000ull) {
    }
  }
  // peers may still write into this CTA's exchange buffers until here
  tc::cluster_sync_all();
}

int launch_fused(int C, const CUtensorMap& mq, const CUtensorMap& mk, const CUtensorMap& mkt,
                 const Stage2TcParams& q, int nclusters, cudaStream_t st) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)(nclusters * C));
  cfg.blockDim = dim3(s2f::THREADS);
  cfg.dynamicSmemBytes = s2_fused_smem_bytes(C);
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  // the register split inside the kernel needs the launch to reserve at least
  // REG_NEEDED registers per CTA; refuse rather than launch a kernel whose
  // setmaxnreg.inc could never be satisfied
  cudaFuncAttributes fa;
  if ((C == 8 ? cudaFuncGetAttributes(&fa, s2_fused_kernel<8>) : cudaFuncGetAttributes(&fa, s2_fused_kernel<4>)) !=
      cudaSuccess)
    return 1;
  if (fa.numRegs * s2f::THREADS < s2f::REG_NEEDED) return 2;
  cudaError_t e;
  if (C == 8) {
    cudaFuncSetAttribute(s2_fused_kernel<8>, cudaFuncAttributeMaxDynamicSharedMemorySize, s2_fused_smem_bytes(8));
    e = cudaLaunchKernelEx(&cfg, s2_fused_kernel<8>, mq, mk, mkt, q);
  } else {
    cudaFuncSetAttribute(s2_fused_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize, s2_fused_smem_bytes(4));
    e = cudaLaunchKernelEx(&cfg, s2_fused_kernel<4>, mq, mk, mkt, q);
  }
  return e == cudaSuccess ? 0 : 1;
}

}  // namespace occam
