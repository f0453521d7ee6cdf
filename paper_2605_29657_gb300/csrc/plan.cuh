// plan.cuh -- the Stage-II work plan (internal header): which Stage-II path
// each sample takes and the item lists of those paths. Run by one CTA (the
// last Stage-I finalize CTA to finish) once every sample's S1 size n1[b] is
// known.
#pragma once

#include "common.cuh"
#include "kernels.cuh"

namespace occam {

// Routes every sample (the fused tensor-core kernel with 4-, 8- or 16-CTA
// clusters where its S1 keys and text keys fit, else the two-pass kernels)
// and writes the item lists, the per-sample item and partial-slot offsets,
// and the item counts. blockDim.x threads, tmp: >= 40 ints of shared memory.
// The two-pass kernels get per-sample item offsets, not item lists.
__device__ __forceinline__ void plan_stage2(const Stage2Params& p, int* tmp) {
  const int tid = threadIdx.x;
  const int nhg = (p.H + kHeadGroup - 1) / kHeadGroup;
  int runA = 0, runB = 0, runF = 0, runF8 = 0, runF16 = 0, runS = 0, runHS = 0;
  // A small batch leaves most SMs idle with 4-CTA clusters: when every text
  // tile of the batch can run at once as a resident 16- (or 8-) CTA cluster,
  // samples take the wider cluster, whose CTAs hold fewer keys and finish
  // each head sooner.
  int wide = 0, hsg = 1;  // hsg: head groups of a split tile (1: no split)
  // the first blockDim.x samples' text lengths and S1 sizes, loaded together
  // up front (one memory round trip instead of two in a row)
  int M0 = 0, n10 = 0;
  if (tid < p.bt.B) {
    M0 = (int)(p.bt.text_off[tid + 1] - p.bt.text_off[tid]);
    n10 = *((volatile int32_t*)&p.n1[tid]);
  }
  if (p.use_fused) {
    int tiles = 0;
    for (int b = tid; b < p.bt.B; b += blockDim.x)
      tiles += b == tid ? (M0 + 127) / 128 : (int)((p.bt.text_off[b + 1] - p.bt.text_off[b] + 127) / 128);
    int total_tiles;
    block_exclusive_scan(tiles, tmp, &total_tiles);
    wide = total_tiles <= p.res16 ? 16 : total_tiles <= p.res8 ? 8 : 0;
    // head split: a batch of at most kHsMaxTiles tiles whose tiles fit hsg
    // times over as resident 16-CTA clusters splits each 16-CTA tile's heads
    // into hsg groups (whole key groups, at least 4 heads each)
    if (wide == 16 && p.has_ppart && total_tiles <= kHsMaxTiles) {
      const int grp = p.H / p.Hkv;
      for (int g = kHsGroups; g >= 2; g >>= 1) {
        if (total_tiles * g <= p.res16 && p.H % g == 0 && p.H / g >= 4 && (p.H / g) % grp == 0) {
          hsg = g;
          break;
        }
      }
    }
  }
  for (int b0 = 0; b0 < p.bt.B; b0 += blockDim.x) {
    const int bb = b0 + tid;
    int nA = 0, nB = 0, nF = 0, nF8 = 0, nF16 = 0;
    if (bb < p.bt.B) {
      const int M = b0 == 0 ? M0 : (int)(p.bt.text_off[bb + 1] - p.bt.text_off[bb]);
      const int n1 = b0 == 0 ? n10 : *((volatile int32_t*)&p.n1[bb]);
      // the fused tensor-core kernel takes a sample when its S1 keys and its
      // causal text keys fit the cluster's TMEM / shared memory
      const bool w16 = wide == 16 && fused_fits(16, n1, M, p.H);
      const bool w8 = !w16 && wide >= 8 && fused_fits(8, n1, M, p.H);
      const bool fused4 = !w16 && !w8 && p.use_fused && fused_fits(kFusedCluster, n1, M, p.H);
      const bool fused8 = w8 || (!w16 && !fused4 && p.use_fused && fused_fits(8, n1, M, p.H));
      const bool fused16 = w16 || (!fused4 && !fused8 && p.use_fused && fused_fits(16, n1, M, p.H));
      if (fused4) {
        nF = (M + 127) / 128;
      } else if (fused8) {
        nF8 = (M + 127) / 128;
      } else if (fused16) {
        nF16 = (M + 127) / 128 * hsg;
      } else {
        const int nch = (n1 + kKeyChunk - 1) / kKeyChunk;
        nA = (M + kStatsTile - 1) / kStatsTile * nhg * s2_stat_splits(n1, M);
        nB = (M + kTextTile - 1) / kTextTile * nch;
      }
      if (M == 0) {
        set_status(p.status, OCCAM_ERR_INVALID_ARG);
        p.ref2[bb] = 0.f;
        p.tau2[bb] = 0.f;
      }
    }
    const int nS = nF * kFusedSlotsPerItem + nF8 * kFusedSlotsPerItem8 + nF16 / hsg * kFusedSlotsPerItem16 +
                   nB;  // s2(r) partial slots of this sample (a split tile's items share its slots)
    const int nHS = hsg > 1 ? nF16 / hsg : 0;  // this sample's head-split tiles
    // the seven item and slot counts, scanned together
    __shared__ int mtmp[7 * 33];
    const int cnt[7] = {nA, nB, nF, nF8, nF16, nS, nHS};
    int ex[7], tot[7];
    block_exclusive_scan_n<7>(cnt, ex, tot, mtmp);
    const int totA = tot[0], totB = tot[1], totF = tot[2], totF8 = tot[3], totF16 = tot[4], totS = tot[5],
              totHS = tot[6];
    const int offA = runA + ex[0], offB = runB + ex[1], offF = runF + ex[2], offF8 = runF8 + ex[3],
              offF16 = runF16 + ex[4], offS = runS + ex[5], offHS = runHS + ex[6];
    if (bb < p.bt.B) {
      for (int i = 0; i < nF; ++i)
        if (offF + i < p.maxF) p.itemsF[offF + i] = make_int4(bb, i * 128, offS + i * kFusedSlotsPerItem, 0);
      for (int i = 0; i < nF8; ++i)
        if (offF8 + i < p.maxF) p.itemsF8[offF8 + i] = make_int4(bb, i * 128, offS + i * kFusedSlotsPerItem8, 0);
      for (int i = 0; i < nF16; ++i) {
        const int tile = i / hsg, hg = i % hsg;
        const int w = hsg > 1 ? ((offHS + tile) << 8) | (hg << 4) | hsg : 0;
        if (offF16 + i < p.maxF)
          p.itemsF16[offF16 + i] = make_int4(bb, tile * 128, offS + tile * kFusedSlotsPerItem16, w);
      }
      for (int t = 0; t < nHS; ++t)
        if (offHS + t < kHsMaxTiles)
          p.itemsHS[offHS + t] = make_int4(bb, t * 128, offS + t * kFusedSlotsPerItem16, hsg);
      p.itemA_off[bb] = offA;
      p.itemB_off[bb] = offB;
      p.slot_off[bb] = offS;
    }
    runA += totA;
    runB += totB;
    runF += totF;
    runF8 += totF8;
    runF16 += totF16;
    runS += totS;
    runHS += totHS;
  }
  if (tid == 0) {
    p.itemA_off[p.bt.B] = runA;
    p.itemB_off[p.bt.B] = runB;
    p.slot_off[p.bt.B] = runS;
    if (runA > p.maxA || runB > p.maxB || runF > p.maxF || runF8 > p.maxF || runF16 > p.maxF)
      set_status(p.status, OCCAM_ERR_CAPACITY);
    p.counters[CNT_NA] = (int)(runA < p.maxA ? runA : p.maxA);
    p.counters[CNT_NB] = (int)(runB < p.maxB ? runB : p.maxB);
    p.counters[CNT_NF] = (int)(runF < p.maxF ? runF : p.maxF);
    p.counters[CNT_NF8] = (int)(runF8 < p.maxF ? runF8 : p.maxF);
    p.counters[CNT_NF16] = (int)(runF16 < p.maxF ? runF16 : p.maxF);
    p.counters[CNT_NHS] = runHS < kHsMaxTiles ? runHS : kHsMaxTiles;
  }
}

}  // namespace occam
