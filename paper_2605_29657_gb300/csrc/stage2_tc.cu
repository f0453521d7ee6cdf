// stage2_tc.cu -- fused Stage-II scoring on the 5th-generation tensor cores
// (tcgen05 + TMEM), for samples whose S1 fits a 4-, 8- or 16-CTA cluster.
//
// What it computes (Sec. 3.5, Eq. 7; App. A, Eqs. 15-16): for sample b, text
// token j and head h, A_{j,h} = softmax over {S1 rows of b} u {text keys 0..j}
// of q_{j,h} k^T / sqrt(d2); P[j, v] = sum_h A_{j,h}(v); s2(v) = max_j P[j, v] / H
// for visual S1 rows and the registers' sum_j P[j, r] / H for s2(r).
//
// Work item = (sample, tile of 128 text rows), processed by one cluster of C
// CTAs (C = 4; 8 or 16 for samples with more S1 keys). The text rows are the 128
// TMEM lanes; each CTA owns 1/C of the sample's S1 keys and of the causal
// text keys. Per head, a CTA's keys form one block of N <= 256 rows: its S1
// keys (padded to a multiple of 32), then its text keys (padded to 16).
// Warp roles (512 threads):
//   producers (warps 0-2): the block's S1 rows by TMA gather4 (four rows of
//      one 128-byte K-block per copy, straight from K2 by index: pruned rows
//      are never read), its text rows by 16-row TMA boxes, and the head's
//      128 x 128 query tile by TMA, all into the 128-byte-swizzled operand
//      layout; key blocks and query tiles are double-buffered by head;
//   MMA issuer (warp 3): S = Q K^T for the whole block as eight
//      128 x N x 16 tcgen05.mma (bf16 in, fp32 accumulate) into a per-head
//      TMEM buffer E (two buffers, alternating by head);
//   statistics warps (8, two per TMEM lane quadrant, one thread per text
//      row): they split E's pieces (whole 64-column groups of S1 keys without
//      masking, then the partial S1 piece and the causal text keys), turn
//      the S1-key logits into exp2(l - group max) written back over E, keep
//      the maxima in shared memory, and reduce the row's softmax max / sum;
//      the quadrant's two warps merge theirs and post the row's log-sum
//      L = max + log2(sum) to every CTA of the cluster with asynchronous
//      distributed-shared-memory stores that complete on an mbarrier of the
//      receiving CTA (no fences);
//   probability warps (4, one per quadrant): once a head's statistics are
//      done in this CTA and the cluster's log-sums are in, they add
//      exp2(group max - M) / Z * E over the S1-key pieces to the head-summed
//      probabilities P (registers, all of the CTA's S1 keys, the whole item),
//      with sum_r exp2(L_r) = exp2(M) Z, and release E for the MMAs of the
//      head after next.
// After the last head the probability warps reduce their P columns over
// their 32 rows: column max -> s2 (atomicMax on the fp32 bit pattern, exact
// and order-free since P >= 0), register columns -> a partial of s2(r)
// reduced in fixed order.
#include <mutex>

#include "common.cuh"
#include "kernels.cuh"
#include "tc5.cuh"

namespace occam {

namespace s2f {
constexpr int QR = 128;                // text rows per item (TMEM lanes)
constexpr int PMAX = kFusedMaxOwnImg;  // max S1 keys per CTA
constexpr int NPC = PMAX / 32;         // S1-key pieces (32 columns each) per CTA
constexpr int QBYTES = QR * 256;       // one head's query tile: 2 K-blocks x 128 rows x 128 B
constexpr int TXT_BOX = 16;            // text key rows per TMA box (the text-key padding unit)
constexpr int NPROD = 3;               // producer warps (0-2): TMA gathers; warp 3 issues MMAs
constexpr int MMA_WARP = NPROD;
constexpr int S_WARP0 = NPROD + 1;     // warpgroups 1-2: statistics warps, two per TMEM lane quadrant
constexpr int P_WARP0 = S_WARP0 + 8;   // warpgroup 3: probability warps, one per TMEM lane quadrant
constexpr int NPW = kFusedPartialWarps;
constexpr int THREADS = (P_WARP0 + NPW) * 32;
// exchange slots: a peer posts head h + 4 into a slot only after this CTA's
// probability warps finished head h (the chain runs through both CTAs' E buffers)
constexpr int NXS = 4;
// register split: warpgroup 0 (producers + MMA issuer) shrinks to REG_LOW per
// thread, the statistics warps to REG_S, the probability warps (which keep P
// in registers) grow to REG_P; the sum must stay within what the CTA was
// launched with (checked on the host before launch)
constexpr int REG_LOW = 56, REG_S = 104, REG_P = 248;
constexpr int REG_NEEDED = S_WARP0 * 32 * REG_LOW + 8 * 32 * REG_S + NPW * 32 * REG_P;
static_assert(S_WARP0 % 4 == 0 && P_WARP0 % 4 == 0 && NPW == 4, "roles split on warpgroup boundaries");
static_assert(REG_NEEDED <= 65536, "register split exceeds the register file");
constexpr uint32_t TMEM_COLS = 512;
static_assert(2 * kFusedKeyRows4 <= (int)TMEM_COLS && 2 * kFusedKeyRows8 <= (int)TMEM_COLS &&
                  2 * kFusedKeyRows16 <= (int)TMEM_COLS,
              "two E buffers");
static_assert(kFusedKeyRows4 % 32 == 0 && kFusedKeyRows8 % 32 == 0 && kFusedKeyRows16 % 32 == 0 &&
                  kFusedKeyRows4 <= 256,
              "MMA N <= 256");
static_assert(PMAX % 32 == 0, "S1 keys in whole pieces");
constexpr uint64_t kLimitNs = 2000000000ull;

template <int C>
struct Geo {
  static constexpr int KROWS = C == 16 ? kFusedKeyRows16 : C == 8 ? kFusedKeyRows8 : kFusedKeyRows4;  // max MMA N
  static constexpr int KBLK = KROWS * 128;                                  // bytes of one K-block of the key rows
  static constexpr uint32_t XBYTES = C * QR * 4;                            // exchange bytes a CTA receives per head
};

template <int C>
struct Smem {
  uint8_t q[2][QBYTES];
  uint8_t k[2][2 * Geo<C>::KBLK];
  float xch[NXS][C][QR];     // log2 of the row's exp2-sum over the CTA's keys, per (slot, CTA, row)
  float cmx[2][NPC][QR];     // per E buffer: the row max of each S1-key piece its exponentials are relative to
  float2 spart[2][4][32];    // per E buffer and lane quadrant: the second statistics warp's (max, sum)
  int32_t kidx[2][PMAX];
  uint8_t kreg[2][PMAX];
  int32_t next_item[4];  // work item of the cluster's ii-th turn, by ii & 3
  uint64_t kfull[2], kempty[2], qfull[2], qempty[2], efull[2], sdone[2], efree[2], xbar[NXS], iready[2], idone[2],
      inext[4], spb[2][4], mdone;
  uint32_t tmem_base;
  int abort;
  uint32_t issued_q;
};
}  // namespace s2f

static_assert(sizeof(s2f::Smem<16>) + 1024 <= 227 * 1024 && sizeof(s2f::Smem<8>) + 1024 <= 227 * 1024 &&
                  sizeof(s2f::Smem<4>) + 1024 <= 227 * 1024,
              "shared memory per CTA");

int s2_fused_smem_bytes(int C) {
  return (int)(C == 16 ? sizeof(s2f::Smem<16>) : C == 8 ? sizeof(s2f::Smem<8>) : sizeof(s2f::Smem<4>)) + 1024;
}
int s2_fused_threads() { return s2f::THREADS; }

namespace {

struct ItemGeom {
  int b, j0, M, n, img0, own_img, txt0, own_txt, ip, tp, N, slot;
  int h0, h1, nhg, hs_tile;  // heads [h0, h1) of this item; head groups of its tile (1: no split)
  bool fits;
  int64_t rbase, t0;
};

template <int C>
__device__ __forceinline__ ItemGeom item_geom(const Stage2TcParams& p, int4 it, int rank) {
  using namespace s2f;
  ItemGeom g;
  g.b = it.x;
  g.j0 = it.y;
  g.slot = it.z;
  const bool item_ok = in_bounds(g.b >= 0 && g.b < p.bt.B, p.status, kSiteFusedItem);
  if (!item_ok) g.b = 0;
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
  g.ip = (g.own_img + 31) & ~31;
  g.tp = (g.own_txt + 15) & ~15;
  g.N = g.ip + g.tp;
  // the same on every CTA of the cluster (depends on the sample only)
  const int ipmax = (per + 31) & ~31;
  g.fits = ipmax <= PMAX && ipmax + ((per_t + 15) & ~15) <= Geo<C>::KROWS;
  // a bad item (checked builds) is skipped by every role of every CTA alike
  g.fits = g.fits && item_ok && in_bounds(g.j0 >= 0 && g.j0 < g.M, p.status, kSiteFusedItem);
  g.nhg = hs_groups(it.w);
  g.h0 = hs_group(it.w) * p.H / g.nhg;
  g.h1 = (hs_group(it.w) + 1) * p.H / g.nhg;
  g.hs_tile = hs_tile(it.w);
  return g;
}

template <class SM>
__device__ __forceinline__ void fail(SM& sm, int* status) {
  sm.abort = 1;
  set_status(status, OCCAM_ERR_TIMEOUT);
}

// Rank 0 of the cluster takes the next work item from the queue and hands it
// to every CTA of the cluster (the value, then a release arrival on the
// CTA's inext barrier). Dynamic hand-out keeps the clusters busy although
// items differ in cost and not every launched cluster is resident at once.
template <int C, class SM>
__device__ __forceinline__ void hand_out_item(SM& sm, int32_t* queue, int ii) {
  const int idx = atomicAdd(queue, 1);
#pragma unroll
  for (int r = 0; r < C; ++r) tc::st_cluster_u32(&sm.next_item[ii & 3], (uint32_t)r, (uint32_t)idx);
#pragma unroll
  for (int r = 0; r < C; ++r) tc::bar_arrive_remote(&sm.inext[ii & 3], (uint32_t)r);
}

// The cluster's ii-th work item (a queue position; >= the item count ends
// the loop). False if the hand-out did not arrive in time.
template <class SM>
__device__ __forceinline__ bool take_item(SM& sm, int ii, volatile int* abort, int& item) {
  if (!tc::bar_wait(&sm.inext[ii & 3], (ii >> 2) & 1, abort, s2f::kLimitNs, true)) return false;
  item = *reinterpret_cast<volatile int32_t*>(&sm.next_item[ii & 3]);
  return true;
}

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Ties the 32 registers a tcgen05.ld wrote to the preceding wait::ld, so the
// compiler cannot move their first use above it.
__device__ __forceinline__ void reg_fence(uint32_t (&v)[32]) {
  asm volatile(""
               : "+r"(v[0]), "+r"(v[1]), "+r"(v[2]), "+r"(v[3]), "+r"(v[4]), "+r"(v[5]), "+r"(v[6]), "+r"(v[7]),
                 "+r"(v[8]), "+r"(v[9]), "+r"(v[10]), "+r"(v[11]), "+r"(v[12]), "+r"(v[13]), "+r"(v[14]), "+r"(v[15]),
                 "+r"(v[16]), "+r"(v[17]), "+r"(v[18]), "+r"(v[19]), "+r"(v[20]), "+r"(v[21]), "+r"(v[22]), "+r"(v[23]),
                 "+r"(v[24]), "+r"(v[25]), "+r"(v[26]), "+r"(v[27]), "+r"(v[28]), "+r"(v[29]), "+r"(v[30]), "+r"(v[31]));
}

__device__ __forceinline__ void ld_wait(uint32_t (&v)[32]) {
  tc::tmem_wait_ld();
  reg_fence(v);
}

__device__ __forceinline__ void ld_wait64(uint32_t (&v)[64]) {
  tc::tmem_wait_ld();
  asm volatile("" : OCCAM_TC_RW64(v));
}

// Statistics of one thread's row over a 32-column piece of logits already
// loaded into v (warp-collective): cm = max of the first `lim` columns in
// log2 units (-inf if none), a = sum over them of exp2(l * sl2 - cm). v is
// overwritten with the exponentials (0 past lim); with `store` (warp-uniform)
// they are also written back to TMEM at sa (the caller waits for that store
// before another thread reads them).
__device__ __forceinline__ void piece_stats(uint32_t (&v)[32], uint32_t sa, int lim, float sl2, bool store, float& cm,
                                            float& a) {
  if (!__all_sync(0xffffffffu, lim >= 32)) {
    // partial piece (causal text keys, the last S1 piece, padded rows):
    // masked logits become -inf, whose exponential is exactly 0
#pragma unroll
    for (int col = 0; col < 32; ++col) v[col] = col < lim ? v[col] : 0xff800000u;
  }
  float t[11];
#pragma unroll
  for (int i = 0; i < 10; ++i)
    t[i] = tc::fmax3(__uint_as_float(v[3 * i]), __uint_as_float(v[3 * i + 1]), __uint_as_float(v[3 * i + 2]));
  t[10] = fmaxf(__uint_as_float(v[30]), __uint_as_float(v[31]));
  const float mx = fmaxf(tc::fmax3(tc::fmax3(t[0], t[1], t[2]), tc::fmax3(t[3], t[4], t[5]), tc::fmax3(t[6], t[7], t[8])),
                         fmaxf(t[9], t[10]));
  cm = mx * sl2;  // -inf when no column is valid
  const float2 sc = make_float2(sl2, sl2);
  const float o = cm == -INFINITY ? 0.f : -cm;
  const float2 off = make_float2(o, o);
  float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    float2 x = __ffma2_rn(make_float2(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1])), sc, off);
    x.x = tc::ex2(x.x);
    x.y = tc::ex2(x.y);
    acc[i & 3] = __fadd2_rn(acc[i & 3], x);
    v[2 * i] = __float_as_uint(x.x);
    v[2 * i + 1] = __float_as_uint(x.y);
  }
  a = ((acc[0].x + acc[0].y) + (acc[1].x + acc[1].y)) + ((acc[2].x + acc[2].y) + (acc[3].x + acc[3].y));
  if (store) tc::tmem_st32(sa, v);
}

// Statistics of one thread's row over 64 columns (two pieces) that are all
// valid S1 keys: cm = their max in log2 units, a = sum of exp2(l * sl2 - cm);
// the exponentials are written back to TMEM at sa. No masking and no
// branches, so the two pieces' dependency chains interleave.
__device__ __forceinline__ void group_stats(uint32_t (&v)[64], uint32_t sa, float sl2, float& cm, float& a) {
  float t[22];
#pragma unroll
  for (int i = 0; i < 21; ++i)
    t[i] = tc::fmax3(__uint_as_float(v[3 * i]), __uint_as_float(v[3 * i + 1]), __uint_as_float(v[3 * i + 2]));
  t[21] = __uint_as_float(v[63]);
  float u[8];
#pragma unroll
  for (int i = 0; i < 7; ++i) u[i] = tc::fmax3(t[3 * i], t[3 * i + 1], t[3 * i + 2]);
  u[7] = t[21];
  const float mx = fmaxf(tc::fmax3(u[0], u[1], u[2]), tc::fmax3(u[3], u[4], fmaxf(u[5], fmaxf(u[6], u[7]))));
  cm = mx * sl2;
  const float2 sc = make_float2(sl2, sl2);
  const float2 off = make_float2(-cm, -cm);
  float2 acc[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) acc[i] = make_float2(0.f, 0.f);
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    float2 x = __ffma2_rn(make_float2(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1])), sc, off);
    x.x = tc::ex2(x.x);
    x.y = tc::ex2(x.y);
    acc[i & 7] = __fadd2_rn(acc[i & 7], x);
    v[2 * i] = __float_as_uint(x.x);
    v[2 * i + 1] = __float_as_uint(x.y);
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) acc[i] = __fadd2_rn(acc[i], acc[i + 4]);
  acc[0] = __fadd2_rn(__fadd2_rn(acc[0], acc[2]), __fadd2_rn(acc[1], acc[3]));
  a = acc[0].x + acc[0].y;
  tc::tmem_st64(sa, v);
}

// merges a finite piece maximum cm (with its sum a) into the running (m, z)
__device__ __forceinline__ void merge_finite(float& m, float& z, float cm, float a) {
  const bool up = cm > m;  // also when m is still -inf (then e = 0 and z = 0)
  const float e = tc::ex2(up ? m - cm : cm - m);
  z = up ? fmaf(z, e, a) : fmaf(a, e, z);
  m = fmaxf(m, cm);
}

// merges a piece's (cm, a) into the row's running softmax (m, z), log2 units
__device__ __forceinline__ void online_merge(float& m, float& z, float cm, float a) {
  if (cm != -INFINITY) {
    // one exponential: the smaller of the two maxima is rescaled to the larger
    const bool up = cm > m;  // also when m is still -inf (then e = 0 and z = 0)
    const float e = tc::ex2(up ? m - cm : cm - m);
    z = up ? fmaf(z, e, a) : fmaf(a, e, z);
    m = up ? cm : m;
  }
}

// P[col] += f * v[col] over one 32-column piece
__device__ __forceinline__ void p_accum(float (&P)[32], const uint32_t (&v)[32], float f) {
  const float2 ff = make_float2(f, f);
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const float2 r2 = __ffma2_rn(make_float2(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1])), ff,
                                 make_float2(P[2 * i], P[2 * i + 1]));
    P[2 * i] = r2.x;
    P[2 * i + 1] = r2.y;
  }
}

}  // namespace

template <int C>
__global__ void __launch_bounds__(s2f::THREADS, 1)
    s2_fused_kernel(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapK,
                    const __grid_constant__ CUtensorMap mapKt, Stage2TcParams p) {
  using namespace s2f;
  using G = Geo<C>;
  extern __shared__ unsigned char smem_raw[];
  Smem<C>& sm = *reinterpret_cast<Smem<C>*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rank = (int)tc::cluster_rank();
  const int nF = p.counters[C == 16 ? CNT_NF16 : C == 8 ? CNT_NF8 : CNT_NF];
  // no work for this cluster (every CTA of every cluster reads the same
  // count): leave before touching shared memory, TMEM or the cluster. With
  // nF items, the clusters numbered nF and up can never be handed one (at
  // most nF hand-outs succeed and the first nF clusters keep drawing until
  // the queue is empty), so they leave too, freeing their SMs at once.
  if ((int)blockIdx.x / C >= nF) return;
  volatile int* abort = &sm.abort;

  if (tid == 0) {
    for (int i = 0; i < 2; ++i) {
      tc::bar_init(&sm.kfull[i], NPROD * 32);
      tc::bar_init(&sm.kempty[i], 1);
      tc::bar_init(&sm.qfull[i], 1);
      tc::bar_init(&sm.qempty[i], 1);
      tc::bar_init(&sm.efull[i], 1);
      tc::bar_init(&sm.sdone[i], 8);
      tc::bar_init(&sm.efree[i], NPW);
      tc::bar_init(&sm.iready[i], NPROD * 32);
      tc::bar_init(&sm.idone[i], NPW);
    }
    // one local arrival (with the expected byte count) plus the peers'
    // asynchronous stores complete each phase of an exchange slot
    for (int i = 0; i < NXS; ++i) tc::bar_init(&sm.xbar[i], 1);
    for (int i = 0; i < 4; ++i) tc::bar_init(&sm.inext[i], 1);
    for (int i = 0; i < 8; ++i) tc::bar_init(&sm.spb[i >> 2][i & 3], 1);
    tc::bar_init(&sm.mdone, 1);
    sm.abort = 0;
    sm.issued_q = 0;
    tc::bar_fence_init();
    for (int i = 0; i < NXS; ++i) tc::bar_expect_tx(&sm.xbar[i], G::XBYTES);
    tc::prefetch_map(&mapQ);
    tc::prefetch_map(&mapK);
    tc::prefetch_map(&mapKt);
  }
  if (warp == MMA_WARP) tc::tmem_alloc(&sm.tmem_base, TMEM_COLS);
  {
    // key buffers start zeroed: rows past a CTA's keys, which are never
    // loaded, then hold finite values, whose logits the epilogue masks out
    uint4* z4 = reinterpret_cast<uint4*>(&sm.k[0][0]);
    constexpr int n16 = (int)(sizeof(sm.k) / 16);
    for (int i = tid; i < n16; i += THREADS) z4[i] = make_uint4(0u, 0u, 0u, 0u);
    tc::fence_proxy_async();
  }
  tc::fence_before();
  __syncthreads();
  tc::fence_after();
  // peers' barriers must be initialised before anyone stores into them remotely
  tc::cluster_sync_all();
  const uint32_t tmem = sm.tmem_base;
  const int H = p.H;

  if (warp < S_WARP0) {
    // warpgroups 0-1: producers and the MMA issuer give registers back
    tc::setmaxnreg_dec<REG_LOW>();
    if (warp < NPROD) {
      // ---------------------------------------------------------- producers
      // NPROD * 32 threads; piece q (16 bytes) of the key block is row (q >> 4), head
      // slice bytes 16 * (q & 15); it lands at the row's 128-byte line of its
      // K-block with the 16-byte chunk index XOR (row & 7).
      const int pt = tid;
      uint32_t qcnt = 0, kcnt = 0;
      int ii = 0;
      for (;; ++ii) {
        if (rank == 0 && pt == 0) hand_out_item<C>(sm, p.queue, ii);
        int item;
        if (!take_item(sm, ii, abort, item)) { fail(sm, p.status); break; }
        if (item >= nF) break;
        const ItemGeom g = item_geom<C>(p, p.items[item], rank);
        if (!g.fits) continue;
        const int ib = ii & 1;
        if (*abort || !tc::bar_wait(&sm.idone[ib], ((ii >> 1) & 1) ^ 1, abort, kLimitNs)) { fail(sm, p.status); break; }
        for (int i = pt; i < g.own_img; i += NPROD * 32) {
          int row = p.dense[g.rbase + g.img0 + i];
          if (!in_bounds(row >= 0 && row < p.bt.total_rows, p.status, kSiteFusedKeyRow)) row = 0;
          sm.kidx[ib][i] = row;
          sm.kreg[ib][i] = p.role[row];
        }
        tc::bar_arrive(&sm.iready[ib]);
        if (!tc::bar_wait(&sm.iready[ib], (ii >> 1) & 1, abort, kLimitNs)) { fail(sm, p.status); break; }
        const int64_t tbase = g.t0 + g.txt0;
        bool ok = true;
        // grouped-query attention: the group's query heads share one key
        // block, loaded for the group's first head (the ring advances per key
        // head); gi = h's index in its group, hkv = the key head it reads
        for (int h = g.h0, gi = 0, hkv = g.h0 / p.kv_group; h < g.h1 && ok;
             ++h, gi = gi + 1 == p.kv_group ? 0 : gi + 1, hkv += gi == 0) {
          const int kb = kcnt & 1;
          const bool load_keys = gi == 0;
          if (load_keys && !tc::bar_wait(&sm.kempty[kb], ((kcnt >> 1) & 1) ^ 1, abort, kLimitNs)) {
            fail(sm, p.status);
            ok = false;
            break;
          }
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
          // The key block by TMA: S1 rows four at a time (gather4: unit u <
          // 2 * gi4 is rows 4 (u >> 1) .. + 3 of K-block u & 1), then the
          // text rows, which are consecutive, in boxes of TXT_BOX rows (rows
          // past a CTA's keys up to the next four / box are loaded but
          // masked; no other padding row is loaded). Every producer thread
          // arrives once per head, announcing the bytes of its own copies
          // before it issues them.
          if (!load_keys) {
            if (gi == p.kv_group - 1) ++kcnt;
            continue;
          }
          const int gi4 = (g.own_img + 3) >> 2, nbt = (g.own_txt + TXT_BOX - 1) / TXT_BOX;
          const int nu = (gi4 + nbt) * 2;
          uint32_t mine = 0;
          for (int u = pt; u < nu; u += NPROD * 32) mine += u < 2 * gi4 ? 512u : (uint32_t)(TXT_BOX * 128);
          tc::bar_expect_tx(&sm.kfull[kb], mine);
          uint8_t* dst = sm.k[kb];
          for (int u = pt; u < nu; u += NPROD * 32) {
            const int kblk = u & 1;
            if (u < 2 * gi4) {
              // S1 rows straight from K2 by index; rows past the CTA's keys repeat its first
              const int r0 = (u >> 1) * 4;
              int y[4];
#pragma unroll
              for (int i = 0; i < 4; ++i) y[i] = sm.kidx[ib][r0 + i < g.own_img ? r0 + i : 0];
              tc::tma_gather4(dst + kblk * G::KBLK + r0 * 128, &mapK, hkv * 128 + kblk * 64, y[0], y[1], y[2], y[3],
                              &sm.kfull[kb]);
            } else {
              const int t0 = ((u >> 1) - gi4) * TXT_BOX;
              tc::tma_load_2d(dst + kblk * G::KBLK + (g.ip + t0) * 128, &mapKt, hkv * 128 + kblk * 64,
                              (int)(tbase + t0), &sm.kfull[kb]);
            }
          }
          if (gi == p.kv_group - 1) ++kcnt;
        }
        if (!ok) break;
      }
      if (pt == 0) sm.issued_q = qcnt;
    } else {
      // ---------------------------------------------------------- MMA issuer
      if (lane == 0) {
        uint32_t qcnt = 0, kcnt = 0, hk = 0;
        for (int ii = 0; !*abort; ++ii) {
          int item;
          if (!take_item(sm, ii, abort, item)) { fail(sm, p.status); break; }
          if (item >= nF) break;
          const ItemGeom g = item_geom<C>(p, p.items[item], rank);
          if (!g.fits) continue;
          const uint32_t idesc = tc::idesc_bf16(128, g.N > 0 ? g.N : 16);
          bool ok = true;
          for (int h = g.h0, gi = 0; h < g.h1 && ok; ++h, ++hk, gi = gi + 1 == p.kv_group ? 0 : gi + 1) {
            const int qb = qcnt & 1, kb = kcnt & 1, eb = hk & 1;
            // E[eb] is free once head hk - 2 was read out of it
            ok = tc::bar_wait(&sm.qfull[qb], (qcnt >> 1) & 1, abort, kLimitNs);
            if (ok && hk >= 2) ok = tc::bar_wait(&sm.efree[eb], ((hk - 2) >> 1) & 1, abort, kLimitNs);
            // the key block of a group of query heads lands once, before its first head
            if (ok && gi == 0) ok = tc::bar_wait(&sm.kfull[kb], (kcnt >> 1) & 1, abort, kLimitNs);
            if (!ok) {
              fail(sm, p.status);
              break;
            }
            // (the operands arrive by TMA, in the async proxy the MMA reads
            // through: the barrier waits above are all the ordering needed)
            tc::fence_after();
            if (g.N > 0) {
              const uint32_t qa = tc::su32(sm.q[qb]), kbase = tc::su32(sm.k[kb]);
#pragma unroll
              for (int s = 0; s < 8; ++s) {
                const int kblk = s >> 2, kk = s & 3;
                tc::mma_bf16(tmem + eb * G::KROWS, tc::sdesc_sw128(qa + kblk * (QBYTES / 2) + kk * 32),
                             tc::sdesc_sw128(kbase + kblk * G::KBLK + kk * 32), idesc, s > 0 ? 1u : 0u);
              }
            }
            tc::mma_commit(&sm.efull[eb]);
            tc::mma_commit(&sm.qempty[qb]);
            if (gi == p.kv_group - 1) {
              // the group's last query head frees the key block
              tc::mma_commit(&sm.kempty[kb]);
              ++kcnt;
            }
            ++qcnt;
          }
        }
        // every MMA issued by this thread has completed once this barrier flips
        tc::mma_commit(&sm.mdone);
        if (!tc::bar_wait(&sm.mdone, 0, nullptr, kLimitNs)) set_status(p.status, OCCAM_ERR_TIMEOUT);
      }
      __syncwarp();
    }
  } else if (warp < P_WARP0) {
    // ------------------------------------------------------------ statistics warps
    // two warps per TMEM lane quadrant (text rows 32 quad .. 32 quad + 31)
    // share every head's pieces of E: whole 64-column groups of S1 keys
    // alternate between them, then the remaining pieces (the partial S1 piece
    // and the causal text keys). Exponentials of S1 keys go back into E with
    // their maxima in cmx; the second warp hands its (max, sum) to the first,
    // which posts the row's statistics to the whole cluster.
    tc::setmaxnreg_dec<REG_S>();
    const int quad = warp & 3;
    const int half = (warp - S_WARP0) >> 2;
    const int j = quad * 32 + lane;
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    const float sl2 = p.scale_log2;
    uint32_t hk = 0;
    for (int ii = 0;; ++ii) {
      int item = 0;
      if (!__all_sync(0xffffffffu, take_item(sm, ii, nullptr, item))) { fail(sm, p.status); break; }
      if (item >= nF) break;
      const ItemGeom g = item_geom<C>(p, p.items[item], rank);
      if (!g.fits) {
        if (tid == S_WARP0 * 32) set_status(p.status, OCCAM_ERR_UNSUPPORTED);
        continue;
      }
      const bool vrow = g.j0 + j < g.M;
      const int jj = g.j0 + j;
      const int npi = g.ip >> 5;
      // pieces of the quadrant: all S1-key pieces, then the text-key pieces
      // up to the causal limit of its last valid row
      const int jl = min(g.j0 + quad * 32 + 31, g.M - 1);
      const int ntc = max(0, min(g.own_txt, jl + 1 - g.txt0));
      const int np = __any_sync(0xffffffffu, vrow) ? npi + ((ntc + 31) >> 5) : 0;
      const int ngf = np > 0 ? g.own_img >> 6 : 0;  // whole 64-column groups of S1 keys
      // the remaining pieces start with the warp that took fewer groups
      const int k0 = 2 * ngf + ((half + ngf) & 1);
      bool ok = true;
      for (int h = g.h0; h < g.h1; ++h, ++hk) {
        const int eb = hk & 1;
        const uint32_t ebase = tmem + lane_base + eb * G::KROWS;
        if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.efull[eb], (hk >> 1) & 1, nullptr, kLimitNs))) {
          ok = false;
          break;
        }
        tc::fence_after();
        float m = -INFINITY, z = 0.f;
        for (int gi = half; gi < ngf; gi += 2) {
          uint32_t v[64];
          tc::tmem_ld64(ebase + gi * 64, v);
          ld_wait64(v);
          float cm, a;
          group_stats(v, ebase + gi * 64, sl2, cm, a);
          sm.cmx[eb][2 * gi][j] = cm;
          sm.cmx[eb][2 * gi + 1][j] = cm;
          merge_finite(m, z, cm, a);
        }
        for (int k = k0; k < np; k += 2) {
          uint32_t v[32];
          tc::tmem_ld32(ebase + k * 32, v);
          ld_wait(v);
          const bool img = k < npi;
          const int lim = !vrow ? 0 : img ? g.own_img - k * 32 : min(g.own_txt - (k * 32 - g.ip), jj - (g.txt0 + k * 32 - g.ip) + 1);
          float cm, a;
          piece_stats(v, ebase + k * 32, lim, sl2, img, cm, a);
          if (img) sm.cmx[eb][k][j] = cm;
          online_merge(m, z, cm, a);
        }
        tc::tmem_wait_st();
        tc::fence_before();
        __syncwarp();
        if (lane == 0) tc::bar_arrive(&sm.sdone[eb]);
        if (half == 1) {
          // hand this warp's (max, sum) to the quadrant's first warp
          // (one buffer per E buffer: this warp reaches head hk + 2 only
          // after the first warp posted head hk)
          sm.spart[eb][quad][lane] = make_float2(m, z);
          __syncwarp();
          if (lane == 0) tc::bar_arrive(&sm.spb[eb][quad]);
        } else {
          if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.spb[eb][quad], (hk >> 1) & 1, nullptr, kLimitNs))) {
            ok = false;
            break;
          }
          const float2 o = sm.spart[eb][quad][lane];
          online_merge(m, z, o.x, o.y);
          // post the row's log-sum L = m + log2(z) (log2 of the sum of exp2
          // of its logits over this CTA's keys; -inf without keys) to the
          // probability warps of every CTA of the cluster
          const float L = z > 0.f ? m + tc::lg2(z) : -INFINITY;
          const int slot = hk & (NXS - 1);
#pragma unroll
          for (int r = 0; r < C; ++r) tc::st_async_f32(&sm.xch[slot][rank][j], &sm.xbar[slot], (uint32_t)r, L);
        }
      }
      if (!ok) { fail(sm, p.status); break; }
    }
  } else {
    // ------------------------------------------------------------ probability warps
    // warp (quad) keeps P for text rows 32 quad .. 32 quad + 31 over all of
    // this CTA's S1 keys in registers. Per head, once the statistics warps
    // are done with it and the cluster's log-sums are in: P +=
    // exp2(cmx - max) / sum * E over the S1-key pieces; then E is released.
    tc::setmaxnreg_inc<REG_P>();
    const int pw = warp - P_WARP0;
    const int quad = warp & 3;
    const int j = quad * 32 + lane;
    const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
    const float invH = 1.0f / (float)H;
    const bool armer = pw == 0 && lane == 0;  // re-arms the exchange slots of this CTA
    uint32_t hk = 0;
    for (int ii = 0;; ++ii) {
      int item = 0;
      if (!__all_sync(0xffffffffu, take_item(sm, ii, nullptr, item))) { fail(sm, p.status); break; }
      if (item >= nF) break;
      const ItemGeom g = item_geom<C>(p, p.items[item], rank);
      if (!g.fits) continue;
      const int ib = ii & 1;
      if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.iready[ib], (ii >> 1) & 1, nullptr, kLimitNs))) { fail(sm, p.status); break; }
      const bool vrow = g.j0 + j < g.M;
      const bool wvalid = __any_sync(0xffffffffu, vrow);  // warp-uniform: any real text row here
      const int npi = g.ip >> 5;
      float P[NPC][32];
#pragma unroll
      for (int q = 0; q < NPC; ++q)
#pragma unroll
        for (int b2 = 0; b2 < 32; ++b2) P[q][b2] = 0.f;
      bool ok = true;
      for (int h = g.h0; h < g.h1; ++h, ++hk) {
        const int eb = hk & 1;
        const int slot = hk & (NXS - 1);
        if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.sdone[eb], (hk >> 1) & 1, nullptr, kLimitNs))) {
          ok = false;
          break;
        }
        if (!__all_sync(0xffffffffu, tc::bar_wait(&sm.xbar[slot], (hk / NXS) & 1, nullptr, kLimitNs, true))) {
          ok = false;
          break;
        }
        tc::fence_after();
        if (wvalid) {
          // the row's softmax denominator over the whole cluster:
          // sum_r exp2(L_r) = exp2(Mx) * Z
          float Mx = -INFINITY;
#pragma unroll
          for (int r = 0; r < C; ++r) Mx = fmaxf(Mx, sm.xch[slot][r][j]);
          float Z = 0.f;
#pragma unroll
          for (int r = 0; r < C; ++r) {
            const float L = sm.xch[slot][r][j];
            if (L != -INFINITY) Z += tc::ex2(L - Mx);
          }
          // Z >= 1 (the largest term is exp2(0)); hardware reciprocal
          const float invZ = (vrow && Z > 0.f) ? tc::rcp(Z) : 0.f;
          const uint32_t pbase = tmem + lane_base + eb * G::KROWS;
#pragma unroll
          for (int q = 0; q < NPC; ++q) {
            if (q < npi) {
              const float cm = sm.cmx[eb][q][j];
              const float f = (invZ > 0.f && cm != -INFINITY) ? tc::ex2(cm - Mx) * invZ : 0.f;
              uint32_t v[32];
              tc::tmem_ld32(pbase + 32 * q, v);
              ld_wait(v);
              p_accum(P[q], v, f);
            }
          }
        }
        tc::fence_before();
        __syncwarp();
        if (lane == 0) tc::bar_arrive(&sm.efree[eb]);
        // the slot's phase for head hk is complete: arm it for head hk + NXS
        if (armer) tc::bar_expect_tx(&sm.xbar[slot], G::XBYTES);
      }
      if (!ok) { fail(sm, p.status); break; }
      if (g.nhg > 1) {
        // a head group of a split tile: its partial head sums go to the
        // scratch, rows of zeros past the text; the merge kernel reduces them
        float* dst = p.ppart + ((((int64_t)g.hs_tile * kHsGroups + hs_group(p.items[item].w)) * 16 + rank) * kHsRows + j) *
                                   PMAX;
#pragma unroll
        for (int q = 0; q < NPC; ++q) {
          if (q < npi) {
#pragma unroll
            for (int c4 = 0; c4 < 8; ++c4)
              *reinterpret_cast<float4*>(dst + q * 32 + 4 * c4) =
                  vrow && wvalid ? make_float4(P[q][4 * c4], P[q][4 * c4 + 1], P[q][4 * c4 + 2], P[q][4 * c4 + 3])
                                 : make_float4(0.f, 0.f, 0.f, 0.f);
          }
        }
        __syncwarp();
        if (lane == 0) tc::bar_arrive(&sm.idone[ib]);
        continue;
      }
      // ---- column reductions of P over this warp's 32 rows: column max ->
      // s2 (atomicMax), register columns -> this warp's partial of s2(r)
      float regacc = 0.f;
      if (wvalid) {
#pragma unroll
        for (int q = 0; q < NPC; ++q) {
          if (q < npi) {
            const int key = q * 32 + lane;
            const bool live = key < g.own_img;
            const bool is_reg = live && sm.kreg[ib][key];
            const uint32_t regmask = __ballot_sync(0xffffffffu, is_reg);
            // register columns first (few): a warp sum over the rows of each
            float rc = 0.f;
            if (regmask) {
#pragma unroll
              for (int col = 0; col < 32; ++col) {
                if (regmask & (1u << col)) {
                  const float sum = warp_sum_f(vrow ? P[q][col] : 0.f);
                  if (lane == col) rc = sum * invH;
                }
              }
            }
            regacc += warp_sum_f(rc);
            // then the column max, transposed in place: afterwards lane l
            // holds the max of this warp's column l of piece q (31 shuffles)
#pragma unroll
            for (int col = 0; col < 32; ++col) P[q][col] = vrow ? P[q][col] : 0.f;
#pragma unroll
            for (int sft = 16; sft >= 1; sft >>= 1) {
              const bool up = (lane & sft) != 0;
#pragma unroll
              for (int i = 0; i < sft; ++i) {
                const float send = up ? P[q][i] : P[q][i + sft];
                const float keep = up ? P[q][i + sft] : P[q][i];
                P[q][i] = fmaxf(keep, __shfl_xor_sync(0xffffffffu, send, sft));
              }
            }
            if (live && !is_reg) atomicMax(reinterpret_cast<int*>(&p.s2[sm.kidx[ib][key]]), __float_as_int(P[q][0] * invH));
          }
        }
      }
      int last = 0;
      if (lane == 0) {
        const int slot = g.slot + rank * NPW + pw;  // C * NPW slots per item
        if (in_bounds(slot >= 0 && slot < p.slot_off[p.bt.B], p.status, kSiteFusedSlot)) p.refpart[slot] = regacc;
        __threadfence();
        const int nslots = p.slot_off[g.b + 1] - p.slot_off[g.b];
        last = atomicAdd(&p.done[g.b], 1) == nslots - 1;
      }
      if (__shfl_sync(0xffffffffu, last, 0)) {
        // the sample's last partial: ref2 = (sum of the partials) / (R M),
        // lane l taking slots l, l + 32, ... in order, then a fixed tree
        __threadfence();
        const int s0 = p.slot_off[g.b], s1 = p.slot_off[g.b + 1];
        float acc = 0.f;
        for (int i = s0 + lane; i < s1; i += 32) acc += __ldcg(&p.refpart[i]);
        acc = warp_sum_f(acc);
        if (lane == 0) {
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
  pdl_trigger();  // a head-split merge behind this launch may be scheduled
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

// Merge of head-split tiles. CTA (t, rank) of a kHsMaxTiles x 16 grid takes
// tile t's S1 keys of cluster rank `rank`: key column k and row quarter q
// belong to thread q * kFusedMaxOwnImg + k. A thread sums the head groups'
// partials (in group order) for each of its rows (rows q, q + 4, ...), with
// every load of its rows issued before the adds, and keeps their max and
// sum; the four quarters then meet in shared memory in quarter order. The
// column max over the tile's text rows goes to s2; the register columns'
// sums over rows, added over the CTA's columns in a fixed order, fill the
// tile's partial slots of that rank. The sample's last slot writer turns the
// slots into ref2 and tau2 as the fused kernel does.
constexpr int kMergeQ = 4;                            // row quarters per key column
constexpr int kMergeThreads = kMergeQ * kFusedMaxOwnImg;
__global__ void __launch_bounds__(kMergeThreads) s2_merge_kernel(Stage2TcParams p) {
  using namespace s2f;
  constexpr int NW = kFusedMaxOwnImg / 32;
  __shared__ float wsum[NW];
  __shared__ float2 qpart[kMergeQ][kFusedMaxOwnImg];  // (column max, column sum) per row quarter
  __shared__ int s_last;
  const int t = blockIdx.x / 16, rank = blockIdx.x % 16;
  if (t >= p.counters[CNT_NHS]) return;
  const int4 it = p.itemsHS[t];
  const int nhg = it.w;
  const ItemGeom g = item_geom<16>(p, make_int4(it.x, it.y, it.z, 0), rank);
  const int k = threadIdx.x % kFusedMaxOwnImg, q = threadIdx.x / kFusedMaxOwnImg, lane = threadIdx.x & 31;
  const int rows = min(kHsRows, g.M - g.j0);
  const float invH = 1.0f / (float)p.H;
  int row_id = 0;
  bool is_reg = false;
  if (q == 0 && k < g.own_img) {
    row_id = p.dense[g.rbase + g.img0 + k];
    if (!in_bounds(row_id >= 0 && row_id < p.bt.total_rows, p.status, kSiteFusedKeyRow)) row_id = 0;
    is_reg = p.role[row_id] != 0;
  }
  // all of the above comes from the Stage-I finalize kernel; the fused
  // kernel's partials (and its s2 and slot writes) only after it finished
  pdl_wait();
  float cmax = 0.f, rsum = 0.f;
  if (k < g.own_img) {
    const float* src = p.ppart + (((int64_t)t * kHsGroups * 16 + rank) * kHsRows) * PMAX + k;
    // this thread's rows q, q + 4, ..., up to eight at a time with every
    // group's load in flight before the adds; sums in group order, then row
    // order
    for (int r0 = q; r0 < rows; r0 += 8 * kMergeQ) {
      float v[8][kHsGroups];
#pragma unroll
      for (int u = 0; u < 8; ++u)
#pragma unroll
        for (int hg = 0; hg < kHsGroups; ++hg) {
          const int r = r0 + u * kMergeQ;
          v[u][hg] = (r < rows && hg < nhg) ? __ldcg(src + ((int64_t)hg * 16 * kHsRows + r) * PMAX) : 0.f;
        }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        if (r0 + u * kMergeQ < rows) {
          float x = v[u][0];
#pragma unroll
          for (int hg = 1; hg < kHsGroups; ++hg) x += v[u][hg];
          cmax = fmaxf(cmax, x);
          rsum += x;
        }
      }
    }
  }
  qpart[q][k] = make_float2(cmax, rsum);
  __syncthreads();
  float rc = 0.f;
  if (q == 0) {
    if (k < g.own_img) {
      float cm = qpart[0][k].x, rs = qpart[0][k].y;
#pragma unroll
      for (int qq = 1; qq < kMergeQ; ++qq) {
        cm = fmaxf(cm, qpart[qq][k].x);
        rs += qpart[qq][k].y;
      }
      if (is_reg) {
        rc = rs * invH;
      } else {
        atomicMax(reinterpret_cast<int*>(&p.s2[row_id]), __float_as_int(cm * invH));
      }
    }
    rc = warp_sum_f(rc);
    if (lane == 0) wsum[k >> 5] = rc;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float acc = 0.f;
    for (int w = 0; w < NW; ++w) acc += wsum[w];
    // the tile's NPW slots of this rank: the sum in the first, zeros after
    p.refpart[g.slot + rank * NPW] = acc;
    for (int i = 1; i < NPW; ++i) p.refpart[g.slot + rank * NPW + i] = 0.f;
    __threadfence();
    const int nslots = p.slot_off[g.b + 1] - p.slot_off[g.b];
    s_last = atomicAdd(&p.done[g.b], NPW) == nslots - NPW;
  }
  __syncthreads();
  if (s_last && threadIdx.x < 32) {
    // the sample's last partials: ref2 = (sum of the partials) / (R M),
    // lane l taking slots l, l + 32, ... in order, then a fixed tree
    __threadfence();
    const int s0 = p.slot_off[g.b], s1 = p.slot_off[g.b + 1];
    float acc = 0.f;
    for (int i = s0 + lane; i < s1; i += 32) acc += __ldcg(&p.refpart[i]);
    acc = warp_sum_f(acc);
    if (lane == 0) {
      const int R = p.bt.reg_off[p.bt.seg_first[g.b + 1]] - p.bt.reg_off[p.bt.seg_first[g.b]];
      const float r2 = (R > 0 && g.M > 0) ? acc / ((float)R * (float)g.M) : 0.f;
      p.ref2[g.b] = r2;
      p.tau2[g.b] = p.lambda2 * r2;
    }
  }
}

void launch_s2_merge(const Stage2TcParams& q, cudaStream_t st) {
  if (q.ppart) {
    // launched right behind the 16-CTA fused kernel with programmatic
    // stream serialization: its item, geometry and key-row loads overlap the
    // end of that kernel, and it waits for the partials (pdl_wait)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(kHsMaxTiles * 16);
    cfg.blockDim = dim3(kMergeThreads);
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    cudaLaunchKernelEx(&cfg, s2_merge_kernel, q);
    count_launch();
  }
}

// How many C-CTA clusters of the fused kernel the current device holds at
// once (a cluster must fit in one GPC, so this is below SMs / C), from the
// occupancy API; looked up once per device and cluster size.
int fused_resident_clusters(int C) {
  static std::mutex mu;
  static int cache[64][3] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  const int ci = C == 16 ? 2 : C == 8 ? 1 : 0;
  std::lock_guard<std::mutex> lock(mu);
  if (cache[dev][ci] != 0) return cache[dev][ci] > 0 ? cache[dev][ci] : 0;
  auto kern = C == 16 ? s2_fused_kernel<16> : C == 8 ? s2_fused_kernel<8> : s2_fused_kernel<4>;
  cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, s2_fused_smem_bytes(C));
  if (C == 16) cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)C);
  cfg.blockDim = dim3(s2f::THREADS);
  cfg.dynamicSmemBytes = s2_fused_smem_bytes(C);
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = C;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) {
    cudaGetLastError();
    n = 0;
  }
  cache[dev][ci] = n > 0 ? n : -1;
  return n > 0 ? n : 0;
}

int launch_fused(int C, const CUtensorMap& mq, const CUtensorMap& mk, const CUtensorMap& mkt, const Stage2TcParams& q,
                 int nclusters, cudaStream_t st) {
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
  auto kern = C == 16 ? s2_fused_kernel<16> : C == 8 ? s2_fused_kernel<8> : s2_fused_kernel<4>;
  cudaFuncAttributes fa;
  if (cudaFuncGetAttributes(&fa, kern) != cudaSuccess) return 1;
  if (fa.numRegs * s2f::THREADS < s2f::REG_NEEDED) return 2;
  cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, s2_fused_smem_bytes(C));
  // 16-CTA clusters exceed the portable limit of 8
  if (C == 16) cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kern, mq, mk, mkt, q);
  count_launch();
  return e == cudaSuccess ? 0 : 1;
}

}  // namespace occam
