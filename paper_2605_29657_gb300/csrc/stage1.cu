// stage1.cu -- Stage I of OccamToken (Sec. 3.4): [CLS] or mutual attention
// scores of every visual and register row, the register reference of each
// segment, and the image-adaptive threshold S1 = {v : s1(v) >= lambda1 s1(r)} u {r}
// (Eqs. 4-6; App. A, Eqs. 10-13).
#include <cooperative_groups.h>

#include "common.cuh"
#include "kernels.cuh"

namespace cg = cooperative_groups;

namespace occam {

// ============================================================================
// [CLS] scoring: one thread-block cluster per segment.
//
// The segment's K1 rows are contiguous in HBM (rows x H x D bf16). Each CTA of
// the cluster streams its share of them through a ring of shared-memory
// stages filled by 1-D bulk (TMA) copies, computes the H per-head logits of
// every row against the segment's [CLS] query, and keeps them in shared
// memory. The per-head softmax max / sum are combined across the cluster
// through distributed shared memory, after which every CTA writes the
// head-averaged probability s1 of its rows. HBM is read exactly once.
// ============================================================================
namespace cls {
constexpr int H = 16, D = 64;
constexpr int kThreads = 256;
constexpr int kRowBytes = H * D * 2;            // 2048
constexpr int kTileRows = 16;                   // rows per stage
constexpr int kStageBytes = kTileRows * kRowBytes;
constexpr int kStages = 2;
constexpr int kLS = H + 1;                      // padded logit row stride (bank spread)
constexpr int kSmem = kStages * kStageBytes + kMaxClsRowsPerCta * kLS * 4 + 1024;
}  // namespace cls

__global__ void __launch_bounds__(cls::kThreads) stage1_cls_kernel(Stage1ClsParams p) {
  using namespace cls;
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = (int)cluster.block_rank();
  const int C = (int)cluster.num_blocks();
  const int seg = blockIdx.x / C;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

  extern __shared__ __align__(1024) unsigned char smem[];
  unsigned char* stage = smem;
  float* logits = reinterpret_cast<float*>(smem + kStages * kStageBytes);
  float* misc = logits + kMaxClsRowsPerCta * kLS;        // 1024 B
  uint64_t* bar = reinterpret_cast<uint64_t*>(misc);     // kStages barriers
  float2* stat = reinterpret_cast<float2*>(misc + 16);   // [H] local (max, sum)
  float* gmax = misc + 16 + 2 * H;                       // [H]
  float* ginv = gmax + H;                                // [H]
  float* lcls = ginv + H;                                // [H]

  const int64_t sb = p.bt.seg_off[seg], se = p.bt.seg_off[seg + 1];
  const int n = (int)(se - sb);
  const int chunk = (n + C - 1) / C;
  const int64_t r0 = sb + (int64_t)rank * chunk;
  int nloc = (se - r0 < (int64_t)chunk) ? (int)(se - r0) : chunk;
  if (nloc < 0) nloc = 0;
  if (nloc > kMaxClsRowsPerCta) {  // host validation prevents this
    if (tid == 0) set_status(p.status, OCCAM_ERR_UNSUPPORTED);
    nloc = 0;
  }
  const int ntiles = (nloc + kTileRows - 1) / kTileRows;

  // lane layout for the dot products: 8 lanes share one (row, head); lane
  // k = lane & 7 owns dims [8k, 8k+8) of that head.
  const int slot = warp * 4 + (lane >> 3);   // 0..31
  const int my_h = slot & (H - 1);
  const int my_rr = slot >> 4;               // 0..1: row parity inside a step
  const int kv = lane & 7;
  float q[8];
  {
    const __nv_bfloat16* qp = p.q_cls + ((int64_t)seg * H + my_h) * D + kv * 8;
    uint4 raw = *reinterpret_cast<const uint4*>(qp);
    const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) { q[2 * i] = bf16_lo(w[i]); q[2 * i + 1] = bf16_hi(w[i]); }
  }

  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) mbar_init(&bar[i], 1);
    fence_mbar_init();
  }
  __syncthreads();
  const unsigned char* gsrc = reinterpret_cast<const unsigned char*>(p.K1) + r0 * kRowBytes;
  if (tid == 0) {
    for (int i = 0; i < kStages && i < ntiles; ++i) {
      const int rows = min(kTileRows, nloc - i * kTileRows);
      mbar_arrive_expect_tx(&bar[i], rows * kRowBytes);
      bulk_g2s(stage + i * kStageBytes, gsrc + (int64_t)i * kStageBytes, rows * kRowBytes, &bar[i]);
    }
  }

  bool timed_out = false;
  int fail_it = 0;
  int issued = min(kStages, ntiles);
  for (int it = 0; it < ntiles; ++it) {
    const int st = it % kStages;
    if (!mbar_wait(&bar[st], (it / kStages) & 1, kSpinLimit)) { timed_out = true; }
    if (__syncthreads_or(timed_out)) { timed_out = true; fail_it = it; break; }
    const unsigned char* buf = stage + st * kStageBytes;
    const int rows = min(kTileRows, nloc - it * kTileRows);
#pragma unroll
    for (int step = 0; step < kTileRows / 2; ++step) {
      const int rr = step * 2 + my_rr;
      float acc = 0.f;
      if (rr < rows) {
        uint4 raw = *reinterpret_cast<const uint4*>(buf + rr * kRowBytes + my_h * D * 2 + kv * 16);
        const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          acc = fmaf(q[2 * i], bf16_lo(w[i]), acc);
          acc = fmaf(q[2 * i + 1], bf16_hi(w[i]), acc);
        }
      }
      acc += __shfl_xor_sync(0xffffffffu, acc, 1);
      acc += __shfl_xor_sync(0xffffffffu, acc, 2);
      acc += __shfl_xor_sync(0xffffffffu, acc, 4);
      if (kv == 0 && rr < rows) logits[(it * kTileRows + rr) * kLS + my_h] = acc * p.scale;
    }
    __syncthreads();
    if (tid == 0 && issued < ntiles) {
      const int rows_n = min(kTileRows, nloc - issued * kTileRows);
      mbar_arrive_expect_tx(&bar[st], rows_n * kRowBytes);
      bulk_g2s(stage + st * kStageBytes, gsrc + (int64_t)issued * kStageBytes, rows_n * kRowBytes,
               &bar[st]);
      ++issued;
    }
  }
  if (timed_out) {
    // Record the failure and drain every copy still in flight (bounded) before
    // the shared memory goes away.
    if (tid == 0) {
      set_status(p.status, OCCAM_ERR_TIMEOUT);
      for (int it = fail_it; it < issued; ++it) mbar_wait(&bar[it % kStages], (it / kStages) & 1, kSpinLimit);
    }
    __syncthreads();
    nloc = 0;
  }

  // [CLS] self key (rank 0 only): l_cls,h = q_h . k_cls,h * scale
  if (tid < H) {
    float l = -INFINITY;
    if (rank == 0 && p.k_cls != nullptr) {
      const __nv_bfloat16* qp = p.q_cls + ((int64_t)seg * H + tid) * D;
      const __nv_bfloat16* kp = p.k_cls + ((int64_t)seg * H + tid) * D;
      float acc = 0.f;
      for (int d = 0; d < D; ++d) acc = fmaf(__bfloat162float(qp[d]), __bfloat162float(kp[d]), acc);
      l = acc * p.scale;
    }
    lcls[tid] = l;
  }
  __syncthreads();

  // local per-head (max, sum of exp): warp w owns heads 2w and 2w+1
  {
    const int h = warp * 2 + (lane >> 4);
    const int sub = lane & 15;
    float m = (sub == 0) ? lcls[h] : -INFINITY;
    for (int r = sub; r < nloc; r += 16) m = fmaxf(m, logits[r * kLS + h]);
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    float z = 0.f;
    if (m != -INFINITY) {
      if (sub == 0 && lcls[h] != -INFINITY) z = expf(lcls[h] - m);
      for (int r = sub; r < nloc; r += 16) z += expf(logits[r * kLS + h] - m);
    }
#pragma unroll
    for (int o = 8; o > 0; o >>= 1) z += __shfl_xor_sync(0xffffffffu, z, o);
    if (sub == 0) stat[h] = make_float2(m, z);
  }
  cluster.sync();
  if (tid < H) {
    float M = -INFINITY;
    for (int r = 0; r < C; ++r) M = fmaxf(M, cluster.map_shared_rank(stat, r)[tid].x);
    float Z = 0.f;
    for (int r = 0; r < C; ++r) {
      const float2 v = cluster.map_shared_rank(stat, r)[tid];
      if (v.y > 0.f) Z += v.y * expf(v.x - M);
    }
    gmax[tid] = M;
    ginv[tid] = 1.0f / Z;
  }
  __syncthreads();
  const float invH = 1.0f / H;
  for (int r = tid; r < nloc; r += kThreads) {
    float s = 0.f;
#pragma unroll
    for (int h = 0; h < H; ++h) s += expf(logits[r * kLS + h] - gmax[h]) * ginv[h];
    p.s1[r0 + r] = s * invH;
    if (p.s2_zero) p.s2_zero[r0 + r] = 0.f;
  }
  cluster.sync();  // peers may still read `stat` through DSMEM until here
}

int stage1_cls_smem_bytes() { return cls::kSmem; }

// ============================================================================
// Stage-I finalize: per segment, the register reference ref1 = mean of s1
// over the segment's registers, the threshold tau1 = lambda1 * ref1, the S1
// mask (registers always in), the row roles, and the order-preserving list
// of the segment's S1 rows. One CTA per segment.
// ============================================================================
__global__ void __launch_bounds__(256) stage1_finalize_kernel(Stage1FinalizeParams p) {
  __shared__ int tmp[40];
  __shared__ float sref;
  const int seg = blockIdx.x;
  const int tid = threadIdx.x;
  const int64_t sb = p.bt.seg_off[seg], se = p.bt.seg_off[seg + 1];
  const int n = (int)(se - sb);
  const int ra = p.bt.reg_off[seg], rb = p.bt.reg_off[seg + 1];
  if (tid == 0) {
    float acc = 0.f;
    if (p.s1)
      for (int i = ra; i < rb; ++i) acc += p.s1[p.bt.reg_idx[i]];
    sref = (rb > ra) ? acc / (float)(rb - ra) : 0.f;
    if (rb <= ra) set_status(p.status, OCCAM_ERR_INVALID_ARG);
    if (p.ref1) p.ref1[seg] = sref;
  }
  // role bytes: 0 visual, 1 register
  for (int r = tid; r < n; r += blockDim.x) p.role[sb + r] = 0;
  __syncthreads();
  for (int i = ra + tid; i < rb; i += blockDim.x) p.role[p.bt.reg_idx[i]] = 1;
  __syncthreads();
  if (!p.do_threshold) return;
  const float tau = p.lambda1 * sref;
  // each thread owns a contiguous run of rows so the list stays in row order
  const int per = (n + blockDim.x - 1) / blockDim.x;
  const int a = min(n, tid * per), z = min(n, a + per);
  int cnt = 0, cvis = 0;
  for (int r = a; r < z; ++r) {
    const bool reg = p.role[sb + r] != 0;
    const bool k = reg || (p.keep_in ? p.keep_in[sb + r] != 0 : p.s1[sb + r] >= tau);
    cnt += k;
    cvis += (k && !reg);
  }
  int total;
  int pos = block_exclusive_scan(cnt, tmp, &total);
  for (int r = a; r < z; ++r) {
    const bool reg = p.role[sb + r] != 0;
    const bool k = reg || (p.keep_in ? p.keep_in[sb + r] != 0 : p.s1[sb + r] >= tau);
    if (p.keep1) p.keep1[sb + r] = k ? 1 : 0;
    if (k) p.s1_list[sb + pos++] = (int32_t)(sb + r);
  }
  int vis_total;
  block_exclusive_scan(cvis, tmp, &vis_total);
  if (tid == 0) {
    p.n1_seg[seg] = total;
    atomicAdd(&p.n1_vis[p.bt.seg_sample[seg]], vis_total);
  }
}

// ============================================================================
// Mutual scoring (Sec. 3.4, Eq. 6): every row u of a segment attends to every
// row v of the segment, per head. Two passes over the keys:
//   pass 1 (mutual_stats_kernel): per query row and head the softmax max and
//          sum over the segment's keys (online, flash-style);
//   pass 2 (mutual_colsum_kernel): per key chunk, sum over all query rows and
//          heads of exp(l - m)/Z, i.e. the attention each key receives.
// Both passes run QK^T on the tensor cores (mma.sync m16n8k16, bf16 in, fp32
// accumulate). d1 is zero-padded to DP (a multiple of 16).
// ============================================================================
namespace mut {
constexpr int kThreads = 128;  // 4 warps x 16 query rows
}

template <int D, int DP>
__device__ __forceinline__ void load_rows_tile(__nv_bfloat16* sdst, const __nv_bfloat16* base,
                                               int64_t row0, int nrows_valid, int nrows_tile,
                                               int row_stride_elems, int head, int tid, int nthreads) {
  // copies rows [row0, row0+nrows_tile) of head `head` into sdst[r][0..DP) (row
  // stride DP+8); rows past nrows_valid and dims past D are zero.
  constexpr int LD = DP + 8;
  constexpr int VPR = DP / 8;  // 16-byte vectors per row
  for (int i = tid; i < nrows_tile * VPR; i += nthreads) {
    const int r = i / VPR, v = i % VPR;
    __nv_bfloat16* dst = sdst + r * LD + v * 8;
    const bool ok = (r < nrows_valid) && (v * 8 < D);
    const __nv_bfloat16* src =
        ok ? base + (row0 + r) * (int64_t)row_stride_elems + (int64_t)head * D + v * 8 : base;
    cp_async16_zfill(dst, src, ok ? 16 : 0);
  }
}

template <int DP, int NT>
__device__ __forceinline__ void warp_qk(float (&S)[NT][4], const __nv_bfloat16* sQ, int q_row0,
                                        const __nv_bfloat16* sK, int k_row0, int lane) {
  constexpr int LD = DP + 8;
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) S[nt][0] = S[nt][1] = S[nt][2] = S[nt][3] = 0.f;
#pragma unroll
  for (int kk = 0; kk < DP / 16; ++kk) {
    uint32_t a[4];
    ldmatrix_x4(a, sQ + (q_row0 + (lane & 7) + ((lane >> 3) & 1) * 8) * LD + kk * 16 + ((lane >> 4) & 1) * 8);
#pragma unroll
    for (int nt = 0; nt < NT; nt += 2) {
      uint32_t b[4];
      ldmatrix_x4(b, sK + (k_row0 + nt * 8 + (lane & 7) + ((lane >> 4) & 1) * 8) * LD + kk * 16 +
                         ((lane >> 3) & 1) * 8);
      mma_bf16_16816(S[nt], a, b[0], b[1]);
      mma_bf16_16816(S[nt + 1], a, b[2], b[3]);
    }
  }
}

template <int D, int DP>
__global__ void __launch_bounds__(mut::kThreads) mutual_stats_kernel(MutualParams p) {
  constexpr int LD = DP + 8;
  constexpr int KT = 64;  // keys per chunk
  __shared__ __align__(128) __nv_bfloat16 sQ[kMutQTile * LD];
  __shared__ __align__(128) __nv_bfloat16 sK[2][KT * LD];
  const int seg = blockIdx.x;
  const int qt = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t sb = p.bt.seg_off[seg], se = p.bt.seg_off[seg + 1];
  const int n = (int)(se - sb);
  const int q0 = qt * kMutQTile;
  if (q0 >= n) return;
  const int nq = min(kMutQTile, n - q0);
  const int HD = p.H * D;
  const float c = p.scale * 1.4426950408889634f;  // log2(e) folded into the scale
  const int nchunks = (n + KT - 1) / KT;
  for (int h = blockIdx.z; h < p.H; h += gridDim.z) {
    load_rows_tile<D, DP>(sQ, p.Q, sb + q0, nq, kMutQTile, HD, h, tid, mut::kThreads);
    load_rows_tile<D, DP>(sK[0], p.K, sb, min(KT, n), KT, HD, h, tid, mut::kThreads);
    cp_async_commit();
    float m[2] = {-INFINITY, -INFINITY}, z[2] = {0.f, 0.f};  // rows g and g+8 (log2 domain max)
    for (int kc = 0; kc < nchunks; ++kc) {
      if (kc + 1 < nchunks) {
        load_rows_tile<D, DP>(sK[(kc + 1) & 1], p.K, sb + (kc + 1) * KT, min(KT, n - (kc + 1) * KT), KT, HD,
                              h, tid, mut::kThreads);
      }
      cp_async_commit();
      cp_async_wait<1>();
      __syncthreads();
      float S[8][4];
      warp_qk<DP, 8>(S, sQ, warp * 16, sK[kc & 1], 0, lane);
      const int kbase = kc * KT;
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        float cm = -INFINITY;
#pragma unroll
        for (int nt = 0; nt < 8; ++nt)
#pragma unroll
          for (int e = 0; e < 2; ++e) {
            const int key = kbase + nt * 8 + (lane & 3) * 2 + e;
            const float x = (key < n) ? S[nt][half * 2 + e] * c : -INFINITY;
            S[nt][half * 2 + e] = x;
            cm = fmaxf(cm, x);
          }
        cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, 1));
        cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, 2));
        const float mn = fmaxf(m[half], cm);
        float acc = 0.f;
#pragma unroll
        for (int nt = 0; nt < 8; ++nt)
#pragma unroll
          for (int e = 0; e < 2; ++e) acc += exp2f(S[nt][half * 2 + e] - mn);
        acc += __shfl_xor_sync(0xffffffffu, acc, 1);
        acc += __shfl_xor_sync(0xffffffffu, acc, 2);
        z[half] = (m[half] == -INFINITY ? 0.f : z[half] * exp2f(m[half] - mn)) + acc;
        m[half] = mn;
      }
      __syncthreads();
    }
    if ((lane & 3) == 0) {
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const int r = warp * 16 + (lane >> 2) + half * 8;
        if (r < nq) p.stats[(sb + q0 + r) * p.H + h] = make_float2(m[half], 1.0f / z[half]);
      }
    }
    __syncthreads();
  }
}

template <int D, int DP>
__global__ void __launch_bounds__(256) mutual_colsum_kernel(MutualParams p) {
  constexpr int LD = DP + 8;
  constexpr int KC = kMutKChunk;  // 128 keys: warp w -> rows (w&3)*16, keys (w>>2)*64
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __nv_bfloat16* sK = reinterpret_cast<__nv_bfloat16*>(smem_raw);            // [2][KC][LD] (by head parity)
  __nv_bfloat16* sQ = sK + 2 * KC * LD;                                      // [2][64][LD]
  float2* sst = reinterpret_cast<float2*>(sQ + 2 * kMutQTile * LD);          // [2][64]
  float* colsum = reinterpret_cast<float*>(sst + 2 * kMutQTile);             // [4][KC]
  const int seg = blockIdx.x;
  const int kc = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int rb = warp & 3, kh = warp >> 2;
  const int64_t sb = p.bt.seg_off[seg], se = p.bt.seg_off[seg + 1];
  const int n = (int)(se - sb);
  const int k0 = kc * KC;
  if (k0 >= n) return;
  const int nk = min(KC, n - k0);
  const int HD = p.H * D;
  const float c = p.scale * 1.4426950408889634f;
  const int nqt = (n + kMutQTile - 1) / kMutQTile;
  float P[8][4];
#pragma unroll
  for (int nt = 0; nt < 8; ++nt) P[nt][0] = P[nt][1] = P[nt][2] = P[nt][3] = 0.f;
  const int njobs = p.H * nqt;  // (head, query tile) pairs, head-major
  auto issue = [&](int job, int buf) {
    const int h = job / nqt, qt = job % nqt;
    if (qt == 0) load_rows_tile<D, DP>(sK + (h & 1) * KC * LD, p.K, sb + k0, nk, KC, HD, h, tid, 256);
    load_rows_tile<D, DP>(sQ + buf * kMutQTile * LD, p.Q, sb + qt * kMutQTile, min(kMutQTile, n - qt * kMutQTile),
                          kMutQTile, HD, h, tid, 256);
    for (int i = tid; i < kMutQTile; i += 256) {
      const int r = qt * kMutQTile + i;
      sst[buf * kMutQTile + i] = (r < n) ? p.stats[(sb + r) * p.H + h] : make_float2(0.f, 0.f);
    }
  };
  issue(0, 0);
  cp_async_commit();
  for (int job = 0; job < njobs; ++job) {
    const int buf = job & 1;
    const int qt = job % nqt;
    const int h = job / nqt;
    if (job + 1 < njobs) issue(job + 1, buf ^ 1);
    cp_async_commit();
    cp_async_wait<1>();
    __syncthreads();
    float S[8][4];
    warp_qk<DP, 8>(S, sQ + buf * kMutQTile * LD, rb * 16, sK + (h & 1) * KC * LD, kh * 64, lane);
    const int rowA = rb * 16 + (lane >> 2);
    const float2 stA = sst[buf * kMutQTile + rowA];
    const float2 stB = sst[buf * kMutQTile + rowA + 8];
    const bool vA = qt * kMutQTile + rowA < n, vB = qt * kMutQTile + rowA + 8 < n;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        if (vA) P[nt][e] += exp2f(fmaf(S[nt][e], c, -stA.x)) * stA.y;
        if (vB) P[nt][2 + e] += exp2f(fmaf(S[nt][2 + e], c, -stB.x)) * stB.y;
      }
    }
    __syncthreads();  // buffers of this job are reused by the loads issued next iteration
  }
  // column sums over the 16 row slots of each warp, then over the 4 row blocks
#pragma unroll
  for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      float v = P[nt][e] + P[nt][2 + e];
      v += __shfl_xor_sync(0xffffffffu, v, 4);
      v += __shfl_xor_sync(0xffffffffu, v, 8);
      v += __shfl_xor_sync(0xffffffffu, v, 16);
      if ((lane >> 2) == 0) colsum[rb * KC + kh * 64 + nt * 8 + (lane & 3) * 2 + e] = v;
    }
  }
  __syncthreads();
  const float norm = 1.0f / ((float)p.H * (float)n);
  for (int k = tid; k < nk; k += 256) {
    const float v = (colsum[k] + colsum[KC + k]) + (colsum[2 * KC + k] + colsum[3 * KC + k]);
    p.s1[sb + k0 + k] = v * norm;
    if (p.s2_zero) p.s2_zero[sb + k0 + k] = 0.f;
  }
}

int mutual_colsum_smem_bytes(int DP) {
  const int LD = DP + 8;
  return (2 * kMutKChunk * LD + 2 * kMutQTile * LD) * 2 + 2 * kMutQTile * 8 + 4 * kMutKChunk * 4;
}

template <int D, int DP>
static void launch_mutual_t(const MutualParams& p, int S_tot, int max_seg_rows, cudaStream_t st) {
  const int qtiles = (max_seg_rows + kMutQTile - 1) / kMutQTile;
  const int kchunks = (max_seg_rows + kMutKChunk - 1) / kMutKChunk;
  const int smem = mutual_colsum_smem_bytes(DP);
  cudaFuncSetAttribute(mutual_colsum_kernel<D, DP>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  mutual_stats_kernel<D, DP><<<dim3(S_tot, qtiles, p.H), mut::kThreads, 0, st>>>(p);
  mutual_colsum_kernel<D, DP><<<dim3(S_tot, kchunks), 256, smem, st>>>(p);
}

void launch_mutual(const MutualParams& p, int d1, int S_tot, int max_seg_rows, cudaStream_t st) {
  if (d1 == 64) launch_mutual_t<64, 64>(p, S_tot, max_seg_rows, st);
  else if (d1 == 72) launch_mutual_t<72, 80>(p, S_tot, max_seg_rows, st);
  else launch_mutual_t<80, 80>(p, S_tot, max_seg_rows, st);
}

// ============================================================================
// Row roles (0 visual, 1 register) from the register lists; the role array
// is zeroed by the caller first.
// ============================================================================
__global__ void roles_scatter_kernel(BatchDev bt, uint8_t* role) {
  const int64_t nreg = bt.reg_off[bt.S_tot];
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nreg; i += (int64_t)gridDim.x * blockDim.x)
    role[bt.reg_idx[i]] = 1;
}

// ============================================================================
// Standalone threshold (Eq. 3): keep[row] for one reference scope.
// ============================================================================
__global__ void __launch_bounds__(256) threshold_kernel(ThresholdParams p) {
  const int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  int vis = 0, samp = -1;
  if (r < p.bt.total_rows) {
    samp = upper_interval(p.bt.row_off, p.bt.B, r);
    bool k;
    if (p.role[r] != 0) {
      k = p.keep_registers != 0;
    } else {
      const int unit = (p.ref_scope == OCCAM_REF_SEGMENT) ? upper_interval(p.bt.seg_off, p.bt.S_tot, r) : samp;
      k = p.s[r] >= p.lambda * p.ref[unit];
      if (p.prev_keep) k = k && (p.prev_keep[r] != 0);
      vis = k ? 1 : 0;
    }
    p.keep[r] = k ? 1 : 0;
  }
  if (p.count_vis) {
    const unsigned grp = __match_any_sync(0xffffffffu, samp);
    const unsigned vb = __ballot_sync(0xffffffffu, vis);
    if ((threadIdx.x & 31) == __ffs(grp) - 1 && samp >= 0) {
      const int c = __popc(vb & grp);
      if (c) atomicAdd(&p.count_vis[samp], c);
    }
  }
}

}  // namespace occam
