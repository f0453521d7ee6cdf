// stage1.cu -- Stage I of OccamToken (Sec. 3.4): [CLS] or mutual attention
// scores of every visual and register row, the register reference of each
// segment, and the image-adaptive threshold S1 = {v : s1(v) >= lambda1 s1(r)} u {r}
// (Eqs. 4-6; App. A, Eqs. 10-13).
#include <mutex>

#include "common.cuh"
#include "kernels.cuh"
#include "plan.cuh"

namespace occam {

// ============================================================================
// [CLS] logits (Sec. 3.4, Eq. 4): l[row][h] = q_cls[seg(row), h] . K1[row, h]
// / sqrt(d1) for every visual and register row, stored in log2 units (times
// log2(e)), so that the finalize kernel's exponentials are plain exp2. The softmax over the
// segment's rows and the head mean are taken by stage1_finalize_kernel from
// these logits (64 bytes per row), so this kernel is a plain stream over K1:
// persistent CTAs each take a contiguous range of 16-row tiles and pull them
// through a ring of shared-memory stages filled by 1-D bulk (TMA) copies.
// HBM is read exactly once.
// ============================================================================
namespace cls {
constexpr int H = 16;
constexpr int kThreads = 256;
constexpr int kTileRows = 16;                   // rows per stage
constexpr int kStages = 3;
template <int D>
struct Geo {
  static constexpr int kRowBytes = H * D * 2;   // 2048 / 2304 / 4096 for d1 = 64 / 72 / 128
  static constexpr int kStageBytes = kTileRows * kRowBytes;
  static constexpr int kSmem = kStages * kStageBytes + 64;
  static constexpr int kLaneDims = D / 8;       // dims of one (row, head) per lane (8 lanes share it)
  static_assert(D % 8 == 0 && kRowBytes % 16 == 0, "rows in whole 16-byte units");
};
static_assert(Geo<128>::kSmem <= 227 * 1024, "shared memory per CTA");

// n consecutive bf16 values as floats: 16-byte loads when the lane's slice is
// a whole number of them, else 2-byte loads (d1 = 72: 9 dims = 18 bytes)
template <int N>
__device__ __forceinline__ void load_bf16(const unsigned char* src, float (&out)[N]) {
  if constexpr (N % 8 == 0) {
#pragma unroll
    for (int c = 0; c < N / 8; ++c) {
      const uint4 raw = *reinterpret_cast<const uint4*>(src + 16 * c);
      const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        out[8 * c + 2 * i] = bf16_lo(w[i]);
        out[8 * c + 2 * i + 1] = bf16_hi(w[i]);
      }
    }
  } else {
#pragma unroll
    for (int i = 0; i < N; ++i) out[i] = __uint_as_float((uint32_t)reinterpret_cast<const uint16_t*>(src)[i] << 16);
  }
}
}  // namespace cls

template <int D>
__global__ void __launch_bounds__(cls::kThreads) stage1_logits_kernel(Stage1ClsParams p) {
  using namespace cls;
  constexpr int kRowBytes = Geo<D>::kRowBytes, kStageBytes = Geo<D>::kStageBytes, NL = Geo<D>::kLaneDims;
  extern __shared__ __align__(128) unsigned char smem[];
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int64_t R = p.bt.total_rows;
  const int64_t nt_all = (R + kTileRows - 1) / kTileRows;
  const int64_t t0 = nt_all * blockIdx.x / gridDim.x;
  const int ntiles = (int)(nt_all * (blockIdx.x + 1) / gridDim.x - t0);
  const unsigned char* gsrc = reinterpret_cast<const unsigned char*>(p.K1);

  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) mbar_init(&bar[i], 1);
    fence_mbar_init();
    for (int i = 0; i < kStages && i < ntiles; ++i) {
      const int64_t r0 = (t0 + i) * kTileRows;
      const int rows = (int)min((int64_t)kTileRows, R - r0);
      mbar_arrive_expect_tx(&bar[i], rows * kRowBytes);
      bulk_g2s(smem + i * kStageBytes, gsrc + r0 * kRowBytes, rows * kRowBytes, &bar[i]);
    }
  }
  __syncthreads();

  // lane layout for the dot products: 8 lanes share one (row, head); lane
  // k = lane & 7 owns dims [k D/8, (k+1) D/8) of that head. The four (row,
  // head) slots of a warp share one row, so segment changes are warp-uniform.
  const int slot = warp * 4 + (lane >> 3);   // 0..31
  const int my_h = slot & (H - 1);
  const int my_rr = slot >> 4;               // 0..1: row parity inside a step
  const int kv = lane & 7;
  int64_t seg_lo = 0, seg_hi = 0;            // rows of the segment q belongs to
  float q[NL];

  bool timed_out = false;
  int it = 0;
  for (; it < ntiles; ++it) {
    const int st = it % kStages;
    // at its last tile the CTA lets the finalize kernel start its input-only
    // prologue (triggered late, so that waiting finalize CTAs do not hold
    // SMs that other work in flight could use)
    if (it == ntiles - 1) pdl_trigger();
    if (!mbar_wait(&bar[st], (it / kStages) & 1, kSpinLimit)) timed_out = true;
    if (__syncthreads_or(timed_out)) {
      timed_out = true;
      break;
    }
    const unsigned char* buf = smem + st * kStageBytes;
    const int64_t r0 = (t0 + it) * kTileRows;
    const int rows = (int)min((int64_t)kTileRows, R - r0);
#pragma unroll
    for (int step = 0; step < kTileRows / 2; ++step) {
      const int rr = step * 2 + my_rr;
      const int64_t row = r0 + rr;
      float acc = 0.f;
      if (rr < rows) {
        if (row >= seg_hi || row < seg_lo) {
          int sg = upper_interval(p.bt.seg_off, p.bt.S_tot, row);
          if (!in_bounds(sg >= 0 && sg < p.bt.S_tot, p.status, kSiteLogitsSegment)) sg = 0;
          seg_lo = p.bt.seg_off[sg];
          seg_hi = p.bt.seg_off[sg + 1];
          load_bf16<NL>(reinterpret_cast<const unsigned char*>(p.q_cls + ((int64_t)sg * H + my_h) * D + kv * NL), q);
        }
        float kx[NL];
        load_bf16<NL>(buf + rr * kRowBytes + my_h * D * 2 + kv * NL * 2, kx);
#pragma unroll
        for (int i = 0; i < NL; ++i) acc = fmaf(q[i], kx[i], acc);
      }
      acc += __shfl_xor_sync(0xffffffffu, acc, 1);
      acc += __shfl_xor_sync(0xffffffffu, acc, 2);
      acc += __shfl_xor_sync(0xffffffffu, acc, 4);
      if (kv == 0 && rr < rows) p.logits[row * H + my_h] = acc * p.scale;  // log2 units
    }
    __syncthreads();
    if (tid == 0 && it + kStages < ntiles) {
      const int64_t rn = (t0 + it + kStages) * kTileRows;
      const int rows_n = (int)min((int64_t)kTileRows, R - rn);
      mbar_arrive_expect_tx(&bar[st], rows_n * kRowBytes);
      bulk_g2s(smem + st * kStageBytes, gsrc + rn * kRowBytes, rows_n * kRowBytes, &bar[st]);
    }
  }
  if (timed_out && tid == 0) {
    // record the failure and drain every copy still in flight (bounded)
    // before the shared memory goes away
    set_status(p.status, OCCAM_ERR_TIMEOUT);
    for (int j = it; j < ntiles && j < it + kStages; ++j) mbar_wait(&bar[j % kStages], (j / kStages) & 1, kSpinLimit);
  }
}

int stage1_logits_smem_bytes(int d1) {
  return d1 == 128 ? cls::Geo<128>::kSmem : d1 == 72 ? cls::Geo<72>::kSmem : cls::Geo<64>::kSmem;
}

void launch_stage1_logits(const Stage1ClsParams& p, int d1, int grid, cudaStream_t st) {
  static std::once_flag once;
  std::call_once(once, [] {
    cudaFuncSetAttribute(stage1_logits_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, cls::Geo<64>::kSmem);
    cudaFuncSetAttribute(stage1_logits_kernel<72>, cudaFuncAttributeMaxDynamicSharedMemorySize, cls::Geo<72>::kSmem);
    cudaFuncSetAttribute(stage1_logits_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         cls::Geo<128>::kSmem);
  });
  const int smem = stage1_logits_smem_bytes(d1);
  if (d1 == 128)
    stage1_logits_kernel<128><<<grid, cls::kThreads, smem, st>>>(p);
  else if (d1 == 72)
    stage1_logits_kernel<72><<<grid, cls::kThreads, smem, st>>>(p);
  else
    stage1_logits_kernel<64><<<grid, cls::kThreads, smem, st>>>(p);
}

// ============================================================================
// Stage-I finalize: per segment, the register reference ref1 = mean of s1
// over the segment's registers, the threshold tau1 = lambda1 * ref1, the S1
// mask (registers always in), the row roles, and the order-preserving list
// of the segment's S1 rows. One CTA per segment.
// ============================================================================
// Merges the softmax statistics of a part into (M, Z, T), all in log2 units:
// M the part's max, Z = sum 2^(x - M), T = sum 2^(x - M) (x - M). A part
// with max -inf is empty.
__device__ __forceinline__ void merge_softmax_stats(float& M, float& Z, float& T, float m2, float z2, float t2) {
  if (m2 == -INFINITY) return;
  if (M == -INFINITY) {
    M = m2;
    Z = z2;
    T = t2;
  } else if (m2 > M) {
    const float d = M - m2, f = fast_exp2(d);
    T = fmaf(f, fmaf(d, Z, T), t2);
    Z = fmaf(Z, f, z2);
    M = m2;
  } else {
    const float d = m2 - M, f = fast_exp2(d);
    T = fmaf(f, fmaf(d, z2, t2), T);
    Z = fmaf(z2, f, Z);
  }
}

// The [CLS] key's own logit per head, l_cls,h = q_cls,h . k_cls,h in log2
// units (-inf without a [CLS] key), into lcls_s[16] (shared): 16 threads per
// head, dims sub, sub + 16, ... It reads only inputs, so it may run before
// the logits kernel has finished. The caller synchronizes before lcls_s is
// read.
__device__ __forceinline__ void cls_self_logits(const Stage1FinalizeParams& p, int seg, float* lcls_s) {
  constexpr int H = 16;
  const int D = p.d1;
  const int tid = threadIdx.x;
  const int hh = tid >> 4, sub = tid & 15;
  float acc = 0.f;
  if (p.k_cls) {
    const __nv_bfloat16* qp = p.q_cls + ((int64_t)seg * H + hh) * D;
    const __nv_bfloat16* kp = p.k_cls + ((int64_t)seg * H + hh) * D;
    for (int d = sub; d < D; d += 16) acc = fmaf(__bfloat162float(qp[d]), __bfloat162float(kp[d]), acc);
  }
#pragma unroll
  for (int o = 8; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (sub == 0) lcls_s[hh] = p.k_cls ? acc * p.scale : -INFINITY;
}

// [CLS] mode (Sec. 3.4, Eq. 4; App. A, Eq. 10): per head h the softmax of the
// [CLS] row over {k_cls} u rows(segment), s1 = mean over heads. The logits
// come in log2 units (the logits kernel scales by log2(e) / sqrt(d1)), so
// 2^(x - max) is each exponential. One pass keeps per thread and head the
// running max, the sum of exponentials and, for the entropy, the sum of
// e (x - max); the block merges them in fixed order; a second pass forms s1
// per row. Both read the logits from global memory (written just before by
// the logits kernel: L2, and L1 for the second pass). s1 is written to s1_out
// (global) and, when given, to s1_loc (shared). lcls_s: the [CLS] key's own
// logit per head (cls_self_logits), in shared memory.
__device__ __forceinline__ void cls_softmax_s1(const Stage1FinalizeParams& p, int seg, int64_t sb, int n,
                                               float* s1_loc, const float* lcls_s) {
  constexpr int H = 16;
  __shared__ float rm[16][17], rz[16][17], rt[16][17];
  __shared__ float gmax[16], ginv[16];
  const int tid = threadIdx.x;
  // thread t takes head (t & 15) of rows (t >> 4) + 16 k: a warp reads 32
  // consecutive floats per row pair. Up to 40 rows' loads are in flight at
  // once, so a segment of up to 640 rows (a 576-token crop with its
  // registers) costs one L2 round trip.
  constexpr int KC = 40;
  const float* lg = p.logits + sb * H;
  const int h = tid & 15, j = tid >> 4;
  float x[KC];
  auto load_chunk = [&](int r0) {
#pragma unroll
    for (int u = 0; u < KC; ++u) {
      const int r = r0 + 16 * u;
      x[u] = r < n ? __ldg(&lg[(int64_t)r * H + h]) : -INFINITY;
    }
  };
  load_chunk(j);
  float m = -INFINITY, z = 0.f, t = 0.f;
  for (int r0 = j;;) {
    float cm = x[0];
#pragma unroll
    for (int u = 1; u < KC; ++u) cm = fmaxf(cm, x[u]);
    if (cm > m) {
      // the running sums move to the new max
      if (m != -INFINITY) {
        const float d = m - cm, f = fast_exp2(d);
        t = f * fmaf(d, z, t);
        z *= f;
      }
      m = cm;
    }
#pragma unroll
    for (int u = 0; u < KC; ++u) {
      const float d = x[u] - m;
      const float e = fast_exp2(d);  // 0 for rows past the segment (-inf)
      z += e;
      t = d > -INFINITY ? fmaf(e, d, t) : t;
    }
    r0 += 16 * KC;
    if (r0 >= n) break;
    load_chunk(r0);
  }
  rm[j][h] = m;
  rz[j][h] = z;
  rt[j][h] = t;
  __syncthreads();
  if (tid < 16) {
    // the [CLS] key itself, then the 16 partials in order
    float M = -INFINITY, Z = 0.f, T = 0.f;
    merge_softmax_stats(M, Z, T, lcls_s[tid], 1.f, 0.f);
    for (int k = 0; k < 16; ++k) merge_softmax_stats(M, Z, T, rm[k][tid], rz[k][tid], rt[k][tid]);
    gmax[tid] = M;
    ginv[tid] = 1.0f / Z;
    // entropy of the head's distribution a = e / Z over the keys:
    // H = -sum a ln a = ln Z - (sum e (l - max)) / Z, with sum e (l - max) =
    // ln 2 * T in log2 units; n_eff = exp(H)
    if (p.n_eff) p.n_eff[(int64_t)seg * H + tid] = expf(logf(Z) - 0.69314718055994531f * T / Z);
  }
  __syncthreads();
  for (int r = tid; r < n; r += blockDim.x) {
    const float4* lp = reinterpret_cast<const float4*>(lg + (int64_t)r * H);
    float acc = 0.f;
#pragma unroll
    for (int k = 0; k < H / 4; ++k) {
      const float4 l = __ldg(lp + k);
      acc += fast_exp2(l.x - gmax[4 * k]) * ginv[4 * k] + fast_exp2(l.y - gmax[4 * k + 1]) * ginv[4 * k + 1] +
             fast_exp2(l.z - gmax[4 * k + 2]) * ginv[4 * k + 2] + fast_exp2(l.w - gmax[4 * k + 3]) * ginv[4 * k + 3];
    }
    const float v = acc * (1.0f / H);
    p.s1_out[sb + r] = v;
    if (s1_loc) s1_loc[r] = v;
    if (p.s2_zero) p.s2_zero[sb + r] = 0.f;
  }
  __syncthreads();
}

// 256 threads, one CTA per segment. With n <= smem_rows the segment's s1
// and roles are staged in shared memory; larger segments work from global
// memory.
__global__ void __launch_bounds__(256) stage1_finalize_kernel(Stage1FinalizeParams p) {
  extern __shared__ float4 fin_smem[];
  __shared__ int tmp[40];
  __shared__ float sref;
  __shared__ int s_seg, s_last;
  __shared__ long long s_base;
  const int tid = threadIdx.x;
  // with S1 lists, segments are taken in ticket order: every earlier segment
  // of the sample has started, so the look-back below always ends
  if (tid == 0) s_seg = p.do_threshold ? atomicAdd(&p.counters[CNT_SEG_TICKET], 1) : (int)blockIdx.x;
  __syncthreads();
  const int seg = s_seg;
  const int64_t sb = p.bt.seg_off[seg], se = p.bt.seg_off[seg + 1];
  const int n = (int)(se - sb);
  const int ra = p.bt.reg_off[seg], rb = p.bt.reg_off[seg + 1];
  // loaded now, used after the softmax: the sample's segment range and row
  // range (for the S1 list) and this thread's first register index
  const int b = p.bt.seg_sample[seg];
  const int s0 = p.bt.seg_first[b], s_next = p.bt.seg_first[b + 1];
  const int64_t row_b = p.bt.row_off[b], row_b1 = p.bt.row_off[b + 1];
  const int64_t reg0 = ra + tid < rb ? (int64_t)p.bt.reg_idx[ra + tid] : -1;
  __shared__ float lcls_s[16];
  if (p.logits) cls_self_logits(p, seg, lcls_s);
  // everything above reads inputs only; what follows reads the previous
  // kernel's results (logits, or s1 in mutual mode)
  pdl_wait();
  const bool staged = n <= p.smem_rows;
  // shared layout for a staged segment: [s1][role]
  float* s1_loc = reinterpret_cast<float*>(fin_smem);
  uint8_t* role_loc = reinterpret_cast<uint8_t*>(s1_loc + p.smem_rows);

  const float* s1g = p.logits ? p.s1_out : p.s1;  // the segment's s1 in global memory
  if (p.logits) {
    cls_softmax_s1(p, seg, sb, n, staged ? s1_loc : nullptr, lcls_s);
  } else if (staged) {
    for (int r = tid; r < n; r += blockDim.x) s1_loc[r] = s1g[sb + r];
  }
  // role bytes: 0 visual, 1 register
  if (staged) {
    for (int r = tid; r < n; r += blockDim.x) role_loc[r] = 0;
    __syncthreads();
    for (int i = ra + tid; i < rb; i += blockDim.x) {
      const int64_t reg = i == ra + tid ? reg0 : p.bt.reg_idx[i];
      if (in_bounds(reg >= sb && reg < se, p.status, kSiteRegisterRow)) role_loc[reg - sb] = 1;
    }
    __syncthreads();
    for (int r = tid; r < n; r += blockDim.x) p.role[sb + r] = role_loc[r];
  } else {
    for (int r = tid; r < n; r += blockDim.x) p.role[sb + r] = 0;
    __syncthreads();
    for (int i = ra + tid; i < rb; i += blockDim.x) {
      const int64_t reg = i == ra + tid ? reg0 : p.bt.reg_idx[i];
      if (in_bounds(reg >= sb && reg < se, p.status, kSiteRegisterRow)) p.role[reg] = 1;
    }
    __syncthreads();
  }
  // ref1 = mean of s1 over the segment's registers (parallel loads, fixed-order
  // sum); under the mean-threshold rule the mean over its visual rows (fp64)
  if (p.ref_mean) {
    const uint8_t* role = staged ? role_loc : p.role + sb;
    double v = 0.0;
    if (s1g)
      for (int r = tid; r < n; r += blockDim.x)
        if (role[r] == 0) v += (double)(staged ? s1_loc[r] : s1g[sb + r]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    __shared__ double dsum[8];
    if ((tid & 31) == 0) dsum[tid >> 5] = v;
    __syncthreads();
    if (tid == 0) {
      double acc = 0.0;
      for (int w = 0; w < (int)(blockDim.x >> 5); ++w) acc += dsum[w];
      const int nv = n - (rb - ra);
      sref = nv > 0 ? (float)(acc / (double)nv) : 0.f;
      if (p.ref1) p.ref1[seg] = sref;
    }
    __syncthreads();
  } else {
    float v = 0.f;
    if (s1g) {
      for (int i = ra + tid; i < rb; i += blockDim.x) {
        const int64_t row = i == ra + tid ? reg0 : p.bt.reg_idx[i];
        v += staged ? s1_loc[row - sb] : s1g[row];
      }
    }
    v = warp_sum(v);
    if ((tid & 31) == 0) tmp[tid >> 5] = __float_as_int(v);
    __syncthreads();
    if (tid == 0) {
      float acc = 0.f;
      for (int w = 0; w < (int)(blockDim.x >> 5); ++w) acc += __int_as_float(tmp[w]);
      sref = (rb > ra) ? acc / (float)(rb - ra) : 0.f;
      if (rb <= ra) set_status(p.status, OCCAM_ERR_INVALID_ARG);
      if (p.ref1) p.ref1[seg] = sref;
    }
    __syncthreads();
  }
  if (!p.do_threshold) return;
  const float tau = p.lambda1 * sref;
  const uint8_t* role = staged ? role_loc : p.role + sb;
  // each thread owns a contiguous run of rows so the list stays in row order
  const int per = (n + blockDim.x - 1) / blockDim.x;
  const int a = min(n, tid * per), z = min(n, a + per);
  int cnt = 0, cvis = 0;
  for (int r = a; r < z; ++r) {
    const bool reg = role[r] != 0;
    const bool k = reg || (p.keep_in ? p.keep_in[sb + r] != 0 : (staged ? s1_loc[r] : s1g[sb + r]) >= tau);
    cnt += k;
    cvis += (k && !reg);
  }
  int total, vis_total;
  int pos = block_exclusive_scan(cnt, tmp, &total);
  block_exclusive_scan(cvis, tmp, &vis_total);
  // this segment's place in its sample's S1 list: a look-back over the
  // sample's earlier segments (warp 0, a window of 32 at a time). A state
  // packs the visual count (bits 31..61) and the key count (bits 0..30)
  // with an "aggregate" or "inclusive prefix" flag.
  constexpr unsigned long long kAgg = 1ull << 62, kPre = 2ull << 62, kLo = (1ull << 31) - 1;
  if (tid < 32) {
    const unsigned long long mine = ((unsigned long long)vis_total << 31) | (unsigned long long)total;
    unsigned long long excl = 0;
    if (seg == s0) {
      if (tid == 0) st_release_u64(&p.seg_state[seg], kPre | mine);
    } else {
      if (tid == 0) st_release_u64(&p.seg_state[seg], kAgg | mine);
      int hi = seg - 1;
      bool timed_out = false;
      uint32_t spins = 0;
      while (true) {
        const int q = hi - tid;
        const unsigned long long v = q >= s0 ? ld_acquire_u64(&p.seg_state[q]) : kPre;
        if (!__all_sync(0xffffffffu, (v & (kAgg | kPre)) != 0)) {
          if (++spins > kSpinLimit) {
            timed_out = true;
            break;
          }
          __nanosleep(32);
          continue;
        }
        const unsigned pre = __ballot_sync(0xffffffffu, (v & kPre) != 0);
        const int first = pre ? __ffs(pre) - 1 : 32;
        unsigned long long val = tid <= first ? (v & ~(kAgg | kPre)) : 0;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) val += __shfl_xor_sync(0xffffffffu, val, o);
        excl += val;
        if (pre) break;
        hi -= 32;
      }
      if (tid == 0) {
        if (timed_out) set_status(p.status, OCCAM_ERR_TIMEOUT);
        st_release_u64(&p.seg_state[seg], kPre | (excl + mine));
      }
    }
    if (tid == 0) {
      s_base = (long long)(excl & kLo);
      if (seg + 1 == s_next) {  // the sample's last segment
        p.n1[b] = (int)((excl & kLo) + (unsigned long long)total);
        if (p.n1_vis) p.n1_vis[b] = (int)(((excl >> 31) & kLo) + (unsigned long long)vis_total);
      }
    }
  }
  __syncthreads();
  int32_t* list = p.dense + row_b + s_base;
  const int64_t list_len = row_b1 - row_b - s_base;  // room left in the sample's list
  for (int r = a; r < z; ++r) {
    const bool reg = role[r] != 0;
    const float sv = p.keep_in ? 0.f : (staged ? s1_loc[r] : s1g[sb + r]);
    const bool k = reg || (p.keep_in ? p.keep_in[sb + r] != 0 : sv >= tau);
    if (p.keep1) p.keep1[sb + r] = k ? 1 : 0;
    // near-threshold flag: the same fp32 tau as the test
    if (p.near1) p.near1[sb + r] = !reg && !p.keep_in && fabsf(sv - tau) <= p.near_rel * fabsf(tau) ? 1 : 0;
    if (k) {
      if (in_bounds(pos >= 0 && pos < list_len, p.status, kSiteListPos)) list[pos] = (int32_t)(sb + r);
      ++pos;
    }
  }
  if (!p.do_plan) return;
  // the last CTA to finish plans Stage II
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = atomicAdd(&p.counters[CNT_DENSE_DONE], 1) == (int)gridDim.x - 1;
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  plan_stage2(p.plan, tmp);
  for (int i = tid; i < p.bt.B; i += blockDim.x) {
    if (p.zero_count_out) p.zero_count_out[i] = 0;
    if (p.zero_count_vis) p.zero_count_vis[i] = 0;
  }
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
