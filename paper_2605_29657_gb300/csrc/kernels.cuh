// kernels.cuh -- kernel parameter blocks and declarations (internal).
#pragma once

#include <cuda.h>

#include "common.cuh"

namespace occam {

constexpr int kFusedCluster = 4;        // CTAs per cluster of the fused tcgen05 Stage-II kernel (C = 8 variant for larger S1)
constexpr int kFusedMaxOwnImg = 192;    // S1 keys one of its CTAs can hold (P columns kept in registers)
constexpr int kFusedKeyRows4 = 256;     // key rows per head one CTA of a 4-CTA cluster holds (= MMA N and TMEM columns)
constexpr int kFusedKeyRows8 = 224;     // the same for an 8-CTA cluster (its exchange buffers take more shared memory)
constexpr int kFusedKeyRows16 = 224;    // and for a 16-CTA cluster (non-portable cluster size)
constexpr int kFusedPartialWarps = 4;   // warps per CTA of the fused kernel that write an s2(r) partial
constexpr int kFinalizeSmemRows = 22400; // Stage-I finalize stages a segment's s1 and roles in shared memory up to this many rows

// Whether a sample with n1 S1 keys and M text tokens fits the fused kernel
// with C CTAs per cluster: each CTA takes ceil(n1 / C) S1 keys (padded to 32)
// and, for the last text tile, ceil(M / C) causal text keys (padded to 16).
// The kernel's item hand-off assumes at least 4 heads per item.
__host__ __device__ inline bool fused_fits(int C, int n1, int M, int H) {
  const int rows = C == 16 ? kFusedKeyRows16 : C == 8 ? kFusedKeyRows8 : kFusedKeyRows4;
  const int ip = ((n1 + C - 1) / C + 31) & ~31;
  const int tp = ((M + C - 1) / C + 15) & ~15;
  return M > 0 && H >= 4 && ip <= kFusedMaxOwnImg && ip + tp <= rows;
}
// Key ranges of the two-pass statistics pass for a sample with n1 S1 keys and
// M text tokens: about four 64-key chunks per range, at most kStatSplits.
// The scores pass merges the ranges' partial statistics, so both passes take
// the count from this one function.
__host__ __device__ inline int s2_stat_splits(int n1, int M) {
  const int s = ((n1 + M + 63) / 64 + 3) / 4;
  return s < 1 ? 1 : s > kStatSplits ? kStatSplits : s;
}
// Head split of small batches: when every text tile of the batch fits as
// kHsGroups resident 16-CTA clusters, each tile's heads are split over that
// many items; their partial head sums meet in a scratch area of kHsMaxTiles
// tiles (allocated only when the batch can have no more tiles than that).
constexpr int kHsMaxTiles = 2;
constexpr int kHsGroups = 8;
constexpr int kHsRows = 128;  // text rows of a fused item
// the fused item's w field: (tile index in the scratch << 8) | (head group << 4) | head groups (0 = 1)
__host__ __device__ inline int hs_groups(int w) { return (w & 15) ? (w & 15) : 1; }
__host__ __device__ inline int hs_group(int w) { return (w >> 4) & 15; }
__host__ __device__ inline int hs_tile(int w) { return w >> 8; }
constexpr int kFusedSlotsPerItem = kFusedCluster * kFusedPartialWarps;  // s2(r) partials per C=4 item
constexpr int kFusedSlotsPerItem8 = 8 * kFusedPartialWarps;             // and per C=8 item
constexpr int kFusedSlotsPerItem16 = 16 * kFusedPartialWarps;           // and per C=16 item

struct Stage1ClsParams {
  BatchDev bt;
  const __nv_bfloat16* q_cls;
  const __nv_bfloat16* K1;
  float scale;  // log2(e) / sqrt(d1): [CLS] logits in log2 units
  float* logits;  // [rows, 16] per-head [CLS] logits in log2 units
  int* status;
};


// Mutual Stage I on the tensor cores (stage1_tc.cu)
struct MutualTcParams {
  BatchDev bt;
  int H;
  int d1;
  float scale_log2;  // log2(e) / sqrt(d1)
  float inv_h;       // 1 / H
  float* lsum;       // [H, total_rows] per query row and head: minus log2 of its softmax denominator (log2 domain)
  float* s1;
  float* s2_zero;    // nullable
  int* status;
  int tiles;         // 128-row tiles of the longest segment
  int32_t* queue;    // [2] work-queue heads of the two passes, zero before the launch
  int hgroups;       // head groups of kMutHeadGroup heads (second pass)
  float* part;       // [hgroups, total_rows] each head group's share of s1
};
constexpr int kMutHeadGroup = 4;


struct ThresholdParams {
  BatchDev bt;
  const float* s;
  const float* ref;
  int ref_scope;
  float lambda;
  const uint8_t* prev_keep;
  int keep_registers;
  const uint8_t* role;
  uint8_t* keep;
  int32_t* count_vis;
};

struct Stage2Params {
  BatchDev bt;
  int H;  // H2, d2 = 128
  int Hkv;  // key / value heads: H, or a divisor of H (grouped-query attention)
  const __nv_bfloat16* Q;   // [total_text, H, 128]
  const __nv_bfloat16* Kt;  // nullable, [total_text, Hkv, 128]
  const __nv_bfloat16* K;   // [rows, Hkv, 128]
  float scale;
  const uint8_t* role;
  int32_t* dense;           // per sample S1 list at row_off[b]
  int32_t* n1;              // [B]
  // two-pass items of sample b are [item*_off[b], item*_off[b + 1]); a
  // kernel finds the sample of its item by binary search and decodes the rest:
  //   stats item i of b:  text tile i / (head groups * key ranges), head group
  //                       (i / key ranges) % head groups, key range i % key ranges
  //   scores item i of b: text tile i / key chunks, key chunk i % key chunks,
  //                       partial slot slot_off[b] + i
  int32_t* itemA_off;       // [B+1]
  int32_t* itemB_off;       // [B+1]
  int32_t* counters;
  int64_t maxA, maxB;
  float2* stats;            // [total_text, H, kStatSplits] partial (max in log2 units, sum) per key range
  float* s2;                // atomicMax accumulator, zeroed beforehand
  float* refpart;           // [maxB]
  int32_t* done;            // [B] finished score items per sample (zeroed)
  int4* itemsF;             // fused items for 4-CTA clusters (b, j0, slot, -)
  int4* itemsF8;            // fused items for 8-CTA clusters
  int4* itemsF16;           // fused items for 16-CTA clusters
  int use_fused;            // route eligible samples to the fused tensor-core kernel
  int res16, res8;          // resident 16- and 8-CTA fused clusters (0: no widening for small batches)
  int4* itemsHS;            // head-split text tiles (b, j0, slot, head groups), for the merge kernel
  int has_ppart;            // the head-split scratch exists
  int32_t* slot_off;        // [B+1] partial-slot range of each sample
  int64_t maxF;
  float* ref2;              // [B]
  float* tau2;              // [B]
  float lambda2;
  int* status;
};

struct Stage1FinalizeParams {
  BatchDev bt;
  // [CLS] mode: the segment's s1 is first formed from the per-head logits
  // (softmax over the segment's rows and the [CLS] self key, head mean)
  const float* logits;            // nullable: s1 is given instead
  const __nv_bfloat16* q_cls;     // [CLS] mode
  const __nv_bfloat16* k_cls;     // nullable
  float scale;  // log2(e) / sqrt(d1): [CLS] logits in log2 units
  int d1 = 64;  // [CLS] mode: head dim of q_cls / k_cls
  float* s1_out;                  // [CLS] mode: where s1 is written
  float* n_eff;                   // nullable, [CLS] mode: [S_tot, 16] effective number of attended keys per head
  float* s2_zero;                 // nullable: zeroed per row (Stage-II max accumulator)
  int smem_rows;                  // segments up to this many rows stage their s1 and roles in shared memory
  uint8_t* near1 = nullptr;       // nullable: near-threshold flags of the Stage-I test
  float near_rel = 1e-5f;         // their relative band
  const float* s1;          // nullable when keep_in is given
  const uint8_t* keep_in;   // nullable: S1 membership of visual rows given instead of tested
  float lambda1;
  int ref_mean;      // 1: ref1 = mean of s1 over the segment's visual rows (mean-threshold rule)
  int do_threshold;
  float* ref1;       // nullable
  uint8_t* role;
  uint8_t* keep1;
  int* status;
  // S1 lists (do_threshold): every sample's S1 rows in row order, at
  // dense[row_off[b]]; segments take their place in the sample's list by a
  // look-back over the sample's earlier segments
  int32_t* dense;
  int32_t* n1;               // [B] S1 keys of the sample (visual + registers)
  int32_t* n1_vis;           // [B] visual S1 rows of the sample
  unsigned long long* seg_state;  // [S_tot] look-back states, zero before the launch
  int32_t* counters;         // CNT_SEG_TICKET, CNT_DENSE_DONE
  // Stage-II work plan, built by the last CTA to finish (do_plan)
  int do_plan;
  Stage2Params plan;
  int32_t* zero_count_out;   // nullable: [B] zeroed by the planning CTA (compaction accumulators)
  int32_t* zero_count_vis;   // nullable
};

struct ScanParams {
  BatchDev bt;
  int mode;                  // 0: keep from `keep_in`; 1: fused Stage-II threshold
  const uint8_t* keep_in;
  const uint8_t* role;
  const uint8_t* keep1;
  const float* s2;
  const float* tau2;
  int keep_registers;
  uint8_t* keep_out;         // nullable
  int64_t capacity;
  int32_t* out_index;
  int32_t* count_out;        // [B] accumulated (zeroed)
  int32_t* count_vis;        // [B] accumulated (zeroed), nullable
  int64_t* out_off;          // [B+1]
  unsigned long long* tile_state;
  int32_t* ticket;
  int64_t ntiles;
  int* status;
  uint8_t* near_out = nullptr;  // nullable, mode 1: near-threshold flags of the Stage-II test
  float near_rel = 1e-5f;       // their relative band
};

struct GatherParams {
  int n_tensors;
  const unsigned char* src[OCCAM_MAX_GATHER];
  unsigned char* dst[OCCAM_MAX_GATHER];
  int64_t row_bytes[OCCAM_MAX_GATHER];
  const int32_t* out_index;
  const int64_t* out_off;    // total kept = out_off[B]
  int B;
  int64_t capacity;
  int64_t src_rows;          // rows of every source tensor (checked builds)
  int* status;               // nullable
};

// Copies the S1 rows of K2 into a staging tensor at the same row positions
// (rows dense[row_off[b] + i], i < n1[b]); the source may be host memory
// the device can read (pinned), the destination is device memory.
struct StageRowsParams {
  BatchDev bt;
  const unsigned char* src;
  unsigned char* dst;
  int64_t row_bytes;
  const int32_t* dense;
  const int32_t* n1;
  int* status;               // nullable
};

// Test-time register construction (Algorithm 1; App. A, register
// redirection): per segment and register channel k, the register rows take
// the max over the visual rows of h[., k], which is then zeroed on them
struct RegistersParams {
  BatchDev bt;
  __nv_bfloat16* h;      // [total_rows, channels]
  int64_t channels;
  const int32_t* k_reg;  // [n_k] channel indices
  int n_k;
  const uint8_t* role;
};

// lambda2 budget matching (App. A): the K-th largest ratio s2[v] / ref2[b(v)]
// over the visual S1 rows of a calibration batch
struct Lambda2Params {
  BatchDev bt;
  const float* s2;
  const float* ref2;
  const uint8_t* keep1;
  const uint8_t* role;
  int64_t target;       // K
  uint32_t* keys;       // [total_rows] scratch
  void* sel;            // kL2SelBytes of zeroed scratch: selection state, histograms, window counts
  float* lambda2;       // out
  int32_t* n_candidates;  // out, nullable
};
constexpr int kL2Digits = 2048;         // lambda2 selection: 11-bit digits
constexpr int kL2Window = 4;            // fp32 steps either way whose kept counts are taken in one pass
constexpr int kL2SelBytes = 32 * 1024;  // workspace scratch of the selection

// mean-threshold reference (component ablation): ref[u] = mean of s over the
// unit's candidate rows (role 0, and prev_keep where given)
struct MeanRefParams {
  BatchDev bt;
  const float* s;
  const uint8_t* role;
  const uint8_t* prev_keep;  // nullable
  int scope;                 // OCCAM_REF_SEGMENT or OCCAM_REF_SAMPLE
  float* ref;                // [units]
  float lambda;
  float* tau;                // nullable: tau[u] = lambda * ref[u]
};

// fixed-budget rule (Sec. 2 top-K; component ablation): per sample the
// budget[b] candidates with the largest s, ties lower row first
struct BudgetParams {
  BatchDev bt;
  const float* s;
  const uint8_t* role;
  const uint8_t* prev_keep;  // nullable
  const int32_t* budget;     // [B]
  int keep_registers;
  uint8_t* keep;             // [total_rows]
  int32_t* count_vis;        // nullable, [B]
};

struct Stage2TcParams {
  BatchDev bt;
  int H;
  float* ppart;             // head-split scratch [kHsMaxTiles][kHsGroups][16][128][kFusedMaxOwnImg]
  const int4* itemsHS;      // head-split tiles (merge kernel)
  int kv_group;             // query heads per key / value head (1 unless grouped-query attention)
  const __nv_bfloat16* K;   // [rows, H / kv_group, 128]
  const __nv_bfloat16* Kt;  // [total_text, H / kv_group, 128] (any valid pointer when has_text == 0)
  float scale_log2;
  int has_text;
  const int32_t* dense;
  const int32_t* n1;
  const uint8_t* role;
  const int4* items;
  const int32_t* counters;
  int32_t* queue;  // item queue head, zero before the launch
  float* s2;
  float* refpart;
  const int32_t* slot_off;
  int32_t* done;
  float* ref2;
  float* tau2;
  float lambda2;
  int* status;
};

// stage1.cu
// the [CLS] logits kernel for d1 = 64, 72 or 128 (stage1.cu)
int stage1_logits_smem_bytes(int d1);
void launch_stage1_logits(const Stage1ClsParams& p, int d1, int grid, cudaStream_t st);
__global__ void stage1_finalize_kernel(Stage1FinalizeParams p);
void launch_mutual_tc(const MutualTcParams& p, const CUtensorMap& mq, const CUtensorMap& mk, const CUtensorMap& mq1,
                      const CUtensorMap& mk1, int sms, cudaStream_t st);
__global__ void roles_scatter_kernel(BatchDev bt, uint8_t* role);
__global__ void threshold_kernel(ThresholdParams p);

// stage2.cu

int s2_stats_smem_bytes();
int launch_stats_tc(const Stage2Params& p, const CUtensorMap& mq128, int grid, cudaStream_t st);

// stage2_tc.cu
int fused_resident_clusters(int C);
void launch_s2_merge(const Stage2TcParams& q, cudaStream_t st);
// stage2_scores_tc.cu
int launch_scores_tc(const Stage2Params& p, const CUtensorMap& mq64, int grid, cudaStream_t st);
int launch_fused(int C, const CUtensorMap& mq, const CUtensorMap& mk, const CUtensorMap& mkt, const Stage2TcParams& q,
                 int nclusters, cudaStream_t st);
int s2_fused_smem_bytes(int C);
int s2_fused_threads();

// compact.cu
__global__ void scan_kernel(ScanParams p);
__global__ void stage_rows_kernel(StageRowsParams p);
__global__ void l2_keys_kernel(Lambda2Params p);
__global__ void l2_hist_kernel(Lambda2Params p, int level);
__global__ void l2_select_kernel(Lambda2Params p, int level);
__global__ void l2_window_kernel(Lambda2Params p);
__global__ void l2_finish_kernel(Lambda2Params p);
__global__ void registers_kernel(RegistersParams p);

// rules.cu
__global__ void mean_ref_kernel(MeanRefParams p);
__global__ void budget_keep_kernel(BudgetParams p);
__global__ void pool_scores_kernel(const float* s_in, int64_t rows_out, int group, int mode, float* s_out);
__global__ void gather_kernel(GatherParams p);
__global__ void offsets_fix_kernel(ScanParams p);

}  // namespace occam
