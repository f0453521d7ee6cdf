// stage2.cu -- Stage II of OccamToken (Sec. 3.5): text-to-vision scores at
// LLM layer l. For sample b and text token j, per head h, the softmax runs
// over the S1 rows of b (visual survivors and registers) and the text keys
// 0..j; p[j, v] is the per-head probability averaged over heads;
// s2(v) = max_j p[j, v], s2(r) = mean over registers and over j (Eq. 7;
// App. A, Eqs. 15-16), and tau2 = lambda2 * s2(r) (Eq. 8).
//
// Work is split in two passes so that any S1 size and any text length fit:
//   stats  (item = sample, 64 text rows, 4 heads, key range): per (j, h)
//          the softmax max and sum over the range's keys, online over
//          64-key chunks; a sample's keys are split into up to 16 ranges so
//          that samples too large for the fused kernel still spread over
//          the SMs;
//   scores (item = sample, 64 text rows, 128 S1 keys): on the 5th-generation
//          tensor cores, in stage2_scores_tc.cu.
// The statistics pass runs QK^T on the tensor cores with mma.sync
// m16n8k16 (bf16 in, fp32 accumulate); its operands are staged in shared
// memory by cp.async.
#include "common.cuh"
#include "kernels.cuh"

namespace occam {

namespace s2k {
constexpr int D = 128;
constexpr int LD = D + 8;  // padded smem row (272 B): conflict-free ldmatrix
constexpr int KT = 64;     // keys per stats chunk
}  // namespace s2k

// copy one 64- or 128-key chunk of query head h's keys into sdst[key][0..128) (stride LD)
__device__ __forceinline__ void s2_load_keys(__nv_bfloat16* sdst, const Stage2Params& p, int b, int64_t t0,
                                             int n_img, int total, int k0, int nkeys_tile, int h, int tid,
                                             int nthreads) {
  using namespace s2k;
  const int64_t rbase = p.bt.row_off[b];
  // grouped-query attention: query head h reads key head h / (H / Hkv)
  const int64_t HD = (int64_t)p.Hkv * D;
  const int64_t hoff = (int64_t)(h / (p.H / p.Hkv)) * D;
  for (int i = tid; i < nkeys_tile * 16; i += nthreads) {
    const int kr = i >> 4, v = i & 15;
    const int kk = k0 + kr;
    const __nv_bfloat16* src = p.K;
    int bytes = 0;
    if (kk < n_img) {
      src = p.K + (int64_t)p.dense[rbase + kk] * HD + hoff + v * 8;
      bytes = 16;
    } else if (kk < total) {
      src = p.Kt + (t0 + (kk - n_img)) * HD + hoff + v * 8;
      bytes = 16;
    }
    cp_async16_zfill(sdst + kr * LD + v * 8, src, bytes);
  }
}

__device__ __forceinline__ void s2_load_queries(__nv_bfloat16* sdst, const Stage2Params& p, int64_t trow0,
                                                int nq, int h, int tid, int nthreads) {
  using namespace s2k;
  const int64_t HD = (int64_t)p.H * D;
  for (int i = tid; i < kTextTile * 16; i += nthreads) {
    const int r = i >> 4, v = i & 15;
    const bool ok = r < nq;
    const __nv_bfloat16* src = ok ? p.Q + (trow0 + r) * HD + (int64_t)h * D + v * 8 : p.Q;
    cp_async16_zfill(sdst + r * LD + v * 8, src, ok ? 16 : 0);
  }
}

// The sample whose items [off[b], off[b + 1]) hold item it (off ascending).
__device__ __forceinline__ int item_sample(const int32_t* off, int B, int it) {
  int lo = 0, hi = B - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (off[mid] <= it) lo = mid; else hi = mid - 1;
  }
  return lo;
}

template <int NT>
__device__ __forceinline__ void warp_qk128(float (&S)[NT][4], const __nv_bfloat16* sQ, int q_row0,
                                           const __nv_bfloat16* sK, int k_row0, int lane) {
  using namespace s2k;
#pragma unroll
  for (int nt = 0; nt < NT; ++nt) S[nt][0] = S[nt][1] = S[nt][2] = S[nt][3] = 0.f;
#pragma unroll
  for (int kk = 0; kk < D / 16; ++kk) {
    uint32_t a[4];
    ldmatrix_x4(a, sQ + (q_row0 + (lane & 7) + ((lane >> 3) & 1) * 8) * LD + kk * 16 + ((lane >> 4) & 1) * 8);
#pragma unroll
    for (int nt = 0; nt < NT; nt += 2) {
      uint32_t bq[4];
      ldmatrix_x4(bq, sK + (k_row0 + nt * 8 + (lane & 7) + ((lane >> 4) & 1) * 8) * LD + kk * 16 +
                          ((lane >> 3) & 1) * 8);
      mma_bf16_16816(S[nt], a, bq[0], bq[1]);
      mma_bf16_16816(S[nt + 1], a, bq[2], bq[3]);
    }
  }
}

// ---------------------------------------------------------------------------
// pass 1: softmax statistics per (text row, head)
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(128) s2_stats_kernel(Stage2Params p) {
  using namespace s2k;
  extern __shared__ __align__(128) unsigned char smem_raw[];
  __nv_bfloat16* sQ = reinterpret_cast<__nv_bfloat16*>(smem_raw);  // [64][LD]
  __nv_bfloat16* sK = sQ + kTextTile * LD;                          // [2][KT][LD]
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nA = p.counters[CNT_NA];
  const float c = p.scale * 1.4426950408889634f;
  for (int it = blockIdx.x; it < nA; it += gridDim.x) {
    const int b = item_sample(p.itemA_off, p.bt.B, it);
    const int64_t t0 = p.bt.text_off[b];
    const int M = (int)(p.bt.text_off[b + 1] - t0);
    const int n_img = p.n1[b];
    const int nhg = (p.H + kHeadGroup - 1) / kHeadGroup;
    const int nsp = s2_stat_splits(n_img, M);
    const int i = it - p.itemA_off[b];
    const int j0 = (i / (nhg * nsp)) * kTextTile, hg = (i / nsp) % nhg, sp = i % nsp;
    const int nq = min(kTextTile, M - j0);
    const int n_txt = p.Kt ? min(j0 + kTextTile, M) : 0;
    const int total = n_img + n_txt;
    // this item's chunks [c0, c1) of the tile's key list (may be empty)
    const int nchunks = (total + KT - 1) / KT;
    const int per = (nchunks + nsp - 1) / nsp;
    const int c0 = min(nchunks, sp * per), c1 = min(nchunks, c0 + per);
    const int jA = j0 + warp * 16 + (lane >> 2), jB = jA + 8;
    const int hend = min(p.H, (hg + 1) * kHeadGroup);
    if (c0 >= c1) {  // an empty key range: neutral partials
      if ((lane & 3) == 0)
        for (int h = hg * kHeadGroup; h < hend; ++h) {
          if (jA < M) p.stats[((t0 + jA) * p.H + h) * kStatSplits + sp] = make_float2(-INFINITY, 0.f);
          if (jB < M) p.stats[((t0 + jB) * p.H + h) * kStatSplits + sp] = make_float2(-INFINITY, 0.f);
        }
      continue;
    }
    for (int h = hg * kHeadGroup; h < hend; ++h) {
      s2_load_queries(sQ, p, t0 + j0, nq, h, tid, 128);
      s2_load_keys(sK, p, b, t0, n_img, total, c0 * KT, KT, h, tid, 128);
      cp_async_commit();
      float m[2] = {-INFINITY, -INFINITY}, z[2] = {0.f, 0.f};
      for (int kc = c0; kc < c1; ++kc) {
        const int lb = (kc - c0) & 1;
        if (kc + 1 < c1) s2_load_keys(sK + (lb ^ 1) * KT * LD, p, b, t0, n_img, total, (kc + 1) * KT, KT, h, tid, 128);
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        float S[8][4];
        warp_qk128<8>(S, sQ, warp * 16, sK + lb * KT * LD, 0, lane);
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          const int j = half ? jB : jA;
          float cm = -INFINITY;
#pragma unroll
          for (int nt = 0; nt < 8; ++nt)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
              const int key = kc * KT + nt * 8 + (lane & 3) * 2 + e;
              const bool valid = key < n_img || (key < total && key - n_img <= j);
              const float x = valid ? S[nt][half * 2 + e] * c : -INFINITY;
              S[nt][half * 2 + e] = x;
              cm = fmaxf(cm, x);
            }
          cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, 1));
          cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, 2));
          const float mn = fmaxf(m[half], cm);
          float acc = 0.f;
          if (mn != -INFINITY) {
#pragma unroll
            for (int nt = 0; nt < 8; ++nt)
#pragma unroll
              for (int e = 0; e < 2; ++e) acc += exp2f(S[nt][half * 2 + e] - mn);
          }
          acc += __shfl_xor_sync(0xffffffffu, acc, 1);
          acc += __shfl_xor_sync(0xffffffffu, acc, 2);
          z[half] = (m[half] == -INFINITY ? 0.f : z[half] * exp2f(m[half] - mn)) + acc;
          m[half] = mn;
        }
        __syncthreads();
      }
      if ((lane & 3) == 0) {
        if (jA < M) p.stats[((t0 + jA) * p.H + h) * kStatSplits + sp] = make_float2(m[0], z[0]);
        if (jB < M) p.stats[((t0 + jB) * p.H + h) * kStatSplits + sp] = make_float2(m[1], z[1]);
      }
    }
  }
}

int s2_stats_smem_bytes() { return (kTextTile + 2 * s2k::KT) * s2k::LD * 2; }

}  // namespace occam
