/*
 * occam.h -- C ABI of the OccamToken prune path on GB300 (sm_103a).
 *
 * OccamToken keeps a visual token v of sample x when its attention score is
 * at least lambda times the score of a test-time register token r that takes
 * part in the same softmax (Sec. 3.2, Eq. 3):
 *
 *   Stage I  (vision encoder):  s1(v) = A_{cls->v} averaged over heads
 *            (Sec. 3.4, Eq. 4; App. A, Eq. 10), or, without [CLS], the mean
 *            attention v receives from all rows (Sec. 3.4, Eq. 6; App. A,
 *            Eq. 13); S1 = {v : s1(v) >= lambda1 s1(r)} u {r} (Eq. 5).
 *   Stage II (LLM layer l):     s2(v) = max_j A_{t_j->v},
 *            s2(r) = mean_j A_{t_j->r} (Sec. 3.5, Eq. 7; App. A, Eqs. 15-16);
 *            S2 = {v in S1\{r} : s2(v) >= lambda2 s2(r)} u {r} (Eq. 8).
 *   Decoding continues on [S2; T] (Algorithm 1), so the kept rows of the
 *   hidden states and of the layer's K/V are compacted (App. A, Eq. 21).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Every pointer argument (except the descriptor structs themselves, the
 *   src/dst/row_bytes arrays of a gather list, and the status out-argument of
 *   occam_get_status) is a DEVICE pointer owned by the caller. The library
 *   allocates no memory: scratch space comes from the caller's `workspace`,
 *   of at least occam_workspace_size() bytes, 256-byte aligned, zero-filled
 *   by the caller before its first use (the library keeps it consistent
 *   afterwards). One workspace serves one call at a time: calls that share
 *   a workspace must be ordered (same stream, or synchronised).
 * - bf16 tensors are dense row-major: [rows, H, d] (K1, Q1, K2),
 *   [segments, H, d] (q_cls, k_cls), [text, H, d] (Q_text, K_text).
 *   Their base addresses must be 16-byte aligned and H*d*2 a multiple of 16.
 * - Rows are numbered sample-major, segment-major: sample b owns rows
 *   [row_off[b], row_off[b+1]), segment s owns rows [seg_off[s], seg_off[s+1]),
 *   segments of one sample are consecutive and tile the sample's rows.
 *   A segment is one encoder pass (an image, a crop, a video frame) with its
 *   own [CLS] query, softmax and registers; register rows are listed per
 *   segment in reg_idx[reg_off[s] .. reg_off[s+1]).
 * - Calls are asynchronous on the caller's stream and never synchronise it.
 *   Host-side argument checks return an error code at once and launch
 *   nothing. Errors found on the device (a capacity overflow, an empty text
 *   query, a bounded wait that ran out) are recorded in a status word inside
 *   the workspace; occam_get_status() reads and clears it.
 * - No C++ exception crosses this boundary.
 */
#ifndef OCCAM_H
#define OCCAM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* occam_stream_t; /* a cudaStream_t; NULL = legacy default stream */

/* Return / status codes. */
enum {
  OCCAM_OK = 0,
  OCCAM_ERR_INVALID_ARG = 1, /* bad size, null pointer, misaligned tensor, M_b = 0, R = 0 */
  OCCAM_ERR_CAPACITY = 2,    /* more kept rows than capacity_rows: rows past capacity are not written */
  OCCAM_ERR_CUDA = 3,        /* a CUDA launch failed (cudaGetLastError) */
  OCCAM_ERR_TIMEOUT = 4,     /* a bounded device-side wait gave up */
  OCCAM_ERR_UNSUPPORTED = 5, /* head count / head dim / size outside what the kernels are built for */
  OCCAM_ERR_WORKSPACE = 6,   /* workspace null, too small or not 256-byte aligned */
  OCCAM_ERR_BOUNDS = 7       /* checked builds (OCCAM_CHECKED=1) only: a computed index fell outside the
                                buffer it addresses; the access was skipped (see occam_get_status) */
};

enum { OCCAM_STAGE1_CLS = 0, OCCAM_STAGE1_MUTUAL = 1 };
enum { OCCAM_REF_SEGMENT = 0, OCCAM_REF_SAMPLE = 1 };
enum { OCCAM_TEXT_KEYS_CAUSAL = 0, OCCAM_TEXT_KEYS_NONE = 1 };
/* Selection rules of occam_prune. REGISTER is the method (Eqs. 5 and 8).
 * MEAN and BUDGET are the variants of the paper's component ablation:
 * MEAN replaces the register score by the mean score of the stage's
 * candidates in both stages; BUDGET keeps Stage I and replaces the Stage-II
 * threshold by a fixed per-sample budget (the top-K rule of Sec. 2). */
enum { OCCAM_RULE_REGISTER = 0, OCCAM_RULE_MEAN = 1, OCCAM_RULE_BUDGET = 2 };
/* Reductions of occam_pool_scores. */
enum { OCCAM_POOL_SUM = 0, OCCAM_POOL_MEAN = 1, OCCAM_POOL_MAX = 2 };

#define OCCAM_MAX_GATHER 8

/* Batch layout. The arrays are device copies; the scalars are host values
 * that must agree with them (they size the launches and the workspace). */
typedef struct occam_batch {
  int32_t B;               /* samples */
  int32_t S_tot;           /* segments over the batch */
  int64_t total_rows;      /* visual + register rows over the batch (< 2^31) */
  int64_t total_text;      /* text tokens over the batch (< 2^31) */
  int32_t max_seg_rows;    /* max rows of one segment */
  int32_t max_sample_rows; /* max rows of one sample */
  int32_t max_text;        /* max text tokens of one sample */
  int32_t max_regs;        /* max registers of one segment */
  const int64_t* row_off;    /* [B+1]   rows of sample b: [row_off[b], row_off[b+1]) */
  const int64_t* seg_off;    /* [S_tot+1] rows of segment s */
  const int32_t* seg_first;  /* [B+1]   segments of sample b: [seg_first[b], seg_first[b+1]) */
  const int32_t* seg_sample; /* [S_tot] sample of segment s */
  const int32_t* reg_idx;    /* [reg_off[S_tot]] global row ids of the register rows */
  const int32_t* reg_off;    /* [S_tot+1] registers of segment s: reg_idx[reg_off[s] .. reg_off[s+1]) */
  const int64_t* text_off;   /* [B+1]   text tokens of sample b: [text_off[b], text_off[b+1]) */
} occam_batch;

/* Stage-I inputs (Sec. 3.4). CLS: q = q_cls [S_tot,H1,d1]; k_cls [S_tot,H1,d1]
 * or NULL (the [CLS] key is then left out of the softmax). MUTUAL: q = Q1
 * [rows,H1,d1], k_cls ignored. K1 [rows,H1,d1]. Built for H1 = 16 with
 * d1 in {64, 72, 128} (CLS) and for 1 <= H1 <= 64 with d1 in {64, 72, 80}
 * (MUTUAL); other shapes return OCCAM_ERR_UNSUPPORTED. */
typedef struct occam_stage1_args {
  int32_t mode; /* OCCAM_STAGE1_CLS or OCCAM_STAGE1_MUTUAL */
  int32_t H1;
  int32_t d1;
  const void* q;
  const void* k_cls;
  const void* K1;
} occam_stage1_args;

/* Stage-II inputs (Sec. 3.5): layer-l queries and keys. Q_text [total_text,H2,d2];
 * K_text [total_text,H2_kv,d2] or NULL (= OCCAM_TEXT_KEYS_NONE: the text keys
 * are left out of the softmax); K2 [rows,H2_kv,d2], read only at S1 rows.
 * Built for d2 = 128 and 1 <= H2 <= 64. */
typedef struct occam_stage2_args {
  int32_t H2;
  int32_t d2;
  const void* Q_text;
  const void* K_text;
  const void* K2;
  /* key / value heads of K2 and K_text: 0 (or H2) for one per query head;
   * a divisor of H2 for grouped-query attention, where query head h reads
   * key head h / (H2 / H2_kv). Rows of K2 and K_text then hold H2_kv * d2
   * values, rows of Q_text H2 * d2. */
  int32_t H2_kv;
} occam_stage2_args;

/* Size of the scratch workspace every entry point needs for this batch and
 * these head counts. Returns OCCAM_OK and writes *bytes. */
int occam_workspace_size(const occam_batch* batch, int32_t H1, int32_t H2, size_t* bytes);

/* Reads and clears the device status word of `workspace` (synchronises
 * `stream`). *status receives OCCAM_OK or the first device-side error code
 * recorded since the last call. In a checked build of the library
 * (compiled with OCCAM_CHECKED=1, every computed index of the kernels'
 * gathers, lists and scans tested against its buffer) a violation records
 * OCCAM_ERR_BOUNDS, and the int32 after the status word (workspace bytes
 * 4..7) names the check site that failed first; both are cleared here. */
int occam_get_status(void* workspace, int32_t* status, occam_stream_t stream);

/* Stage-I scores (Sec. 3.4, Eqs. 4 and 6; App. A, Eqs. 10 and 13).
 * s1 [total_rows] fp32: head-averaged attention each row receives;
 * ref1 [S_tot] fp32: the mean of s1 over the segment's registers (the
 * reference s1(r); with one register it is exactly the paper's). */
int occam_score_stage1(const occam_batch* batch, const occam_stage1_args* args, float* s1,
                       float* ref1, void* workspace, size_t workspace_bytes, occam_stream_t stream);

/* Register-anchored threshold (Eq. 3; Stage I Eq. 5, Stage II Eq. 8).
 * keep[row] = 1 for a visual row with s[row] >= lambda * ref[unit(row)] and
 * (prev_keep == NULL or prev_keep[row] != 0); unit = segment (ref_scope =
 * OCCAM_REF_SEGMENT, ref [S_tot]) or sample (OCCAM_REF_SAMPLE, ref [B]).
 * Register rows are not candidates: keep[reg] = keep_registers.
 * count_vis [B] (int32, may be NULL) receives the kept visual rows per sample. */
int occam_threshold(const occam_batch* batch, const float* s, const float* ref, int32_t ref_scope,
                    float lambda, const uint8_t* prev_keep, int32_t keep_registers, uint8_t* keep,
                    int32_t* count_vis, void* workspace, size_t workspace_bytes, occam_stream_t stream);

/* Mean-threshold reference (component ablation, "Mean threshold"). ref[u]
 * = the mean of s over the candidate rows of unit u: an fp64 sum in a fixed
 * order, divided by the count and rounded to fp32; 0 for a unit without
 * candidates. Candidates are the visual rows with prev_keep[row] != 0
 * (prev_keep NULL: every visual row). unit = segment (ref_scope =
 * OCCAM_REF_SEGMENT, ref [S_tot]) or sample (OCCAM_REF_SAMPLE, ref [B]).
 * occam_threshold with this ref applies the mean-threshold rule. */
int occam_mean_reference(const occam_batch* batch, const float* s, int32_t ref_scope, const uint8_t* prev_keep,
                         float* ref, void* workspace, size_t workspace_bytes, occam_stream_t stream);

/* Fixed-budget selection (Sec. 2, S = top-K(V, s); component ablation,
 * "Fixed budget"). Candidates are the visual rows with prev_keep[row] != 0
 * (prev_keep NULL: every visual row); n_b is sample b's candidate count.
 * In sample b, keep[row] = 1 for the first min(budget[b], n_b) candidates
 * in the order "s high first, then row id low first", so equal scores keep
 * the lower row. budget [B] int32 (device; a negative entry counts as 0).
 * Register rows get keep_registers, every other row 0. count_vis [B]
 * (int32, nullable) receives min(budget[b], n_b). Exact: the decision uses
 * the fp32 values of s. */
int occam_budget_keep(const occam_batch* batch, const float* s, const uint8_t* prev_keep, const int32_t* budget,
                      int32_t keep_registers, uint8_t* keep, int32_t* count_vis, void* workspace,
                      size_t workspace_bytes, occam_stream_t stream);

/* Merged-token scores from patch scores. A 2x2 patch merger (Qwen3-VL's)
 * turns every group of `group` consecutive patch rows into one token; the
 * paper does not say how patch scores become token scores. s_out[i] = the
 * sum (OCCAM_POOL_SUM, the attention mass the group receives), mean
 * (OCCAM_POOL_MEAN) or max (OCCAM_POOL_MAX) of s_in[group i .. group i +
 * group - 1], added in row order. s_in [rows_in], s_out [rows_in / group]
 * fp32, device; rows_in must be a multiple of group (>= 1), else
 * OCCAM_ERR_INVALID_ARG. */
int occam_pool_scores(const float* s_in, int64_t rows_in, int32_t group, int32_t mode, float* s_out,
                      occam_stream_t stream);

/* Stage-II scores (Sec. 3.5, Eq. 7; App. A, Eqs. 15-16). keep1 [total_rows]
 * u8 marks the visual rows of S1 (register rows are always in S1). For
 * sample b and text token j, per head, the softmax runs over the S1 rows of
 * b and the text keys 0..j (causal); the per-head probabilities are averaged
 * over heads. s2 [total_rows] fp32 = max over j for visual S1 rows, 0 for
 * every other row; ref2 [B] fp32 = the mean over the sample's registers of
 * the mean over j. */
int occam_score_stage2(const occam_batch* batch, const occam_stage2_args* args, const uint8_t* keep1,
                       float* s2, float* ref2, void* workspace, size_t workspace_bytes,
                       occam_stream_t stream);

/* Order-preserving stream compaction of the rows with keep[row] != 0
 * (Algorithm 1: decoding continues on [S2; T]). out_index [capacity_rows]
 * int32 receives the kept global row ids in ascending order (hence sample-
 * major), count_out [B] int32 the kept rows per sample and out_off [B+1]
 * int64 their exclusive prefix (out_off[B] = total kept). For each of the
 * n_tensors gather tensors t (0 <= n_tensors <= OCCAM_MAX_GATHER; host arrays
 * of device pointers), row out_off[b]+k of dst[t] becomes an exact copy of
 * the k-th kept row of src[t]; row_bytes[t] is the row size (multiple of 16,
 * pointers 16-byte aligned). If more than capacity_rows rows are kept,
 * nothing is written past capacity_rows, the device status records
 * OCCAM_ERR_CAPACITY, and counts and offsets are still exact. */
int occam_compact(const occam_batch* batch, const uint8_t* keep, int32_t n_tensors,
                  const void* const* src, const int64_t* row_bytes, void* const* dst,
                  int64_t capacity_rows, int32_t* out_index, int32_t* count_out, int64_t* out_off,
                  void* workspace, size_t workspace_bytes, occam_stream_t stream);

/* Test-time register construction (Algorithm 1, step 2; App. A, register
 * redirection), the step before Stage I. h [total_rows, channels] bf16
 * (device, in place) holds the activations of the layer that carries the
 * register neurons; k_reg [n_k] int32 (device) lists those channels,
 * distinct and each in [0, channels) (not checked on the device). For every segment s and k
 * in k_reg: every register row r of s gets h[r][k] = max over the visual
 * rows v of s of h[v][k], and then h[v][k] = 0 on those visual rows. Other
 * channels and rows are unchanged; a segment without visual rows keeps its
 * registers. Exact (the max is one of the inputs). */
int occam_construct_registers(const occam_batch* batch, void* h, int64_t channels, const int32_t* k_reg,
                              int32_t n_k, void* workspace, size_t workspace_bytes, occam_stream_t stream);

/* Budget matching for lambda2 on the device (App. A, lambda2* of the
 * average-budget equation). Over a calibration batch the Stage-II retained
 * count at lambda2 is the number of visual S1 rows v (keep1[v] != 0, not a
 * register) with s2[v] >= lambda2 * ref2[b(v)], so it steps down at each
 * ratio s2[v] / ref2[b(v)]. lambda2_out (device, one fp32) receives the
 * largest fp32 lambda2 under which the test as this library applies it,
 * s2[v] >= fl(lambda2 * ref2[b(v)]) in fp32, keeps at least target_count
 * rows: the target_count-th largest IEEE fp32 quotient s2 / ref2, moved by
 * single fp32 steps where the product's rounding disagrees with the
 * quotient's. Just above it the test keeps fewer rows.
 * target_count = K_tar * |D| in total over the batch's samples. Samples with
 * ref2 <= 0 contribute no candidates. target_count <= 0 gives +inf; a
 * target above the candidate count gives 0 (keep all). n_candidates (device
 * int32, nullable) receives the candidate count. s2 [total_rows] and ref2
 * [B] are as written by occam_score_stage2 / occam_prune. */
int occam_calibrate_lambda2(const occam_batch* batch, const float* s2, const float* ref2, const uint8_t* keep1,
                            int64_t target_count, float* lambda2_out, int32_t* n_candidates, void* workspace,
                            size_t workspace_bytes, occam_stream_t stream);

/* The fused path: Stage-I scores -> Stage-I threshold (per segment,
 * lambda1; registers always in S1) -> Stage-II scores over S1 -> Stage-II
 * threshold (per sample, lambda2) -> compaction and gather. Under the
 * method's rule per-sample budgets are outputs, never inputs (App. A: no
 * hard token budget); only the fixed-budget variant takes them as input. */
typedef struct occam_prune_args {
  occam_batch batch;
  occam_stage1_args stage1;
  occam_stage2_args stage2;
  float lambda1;
  float lambda2;
  int32_t keep_registers; /* 1: register rows are emitted (the paper keeps r); 0: visual rows only */
  int32_t n_tensors;      /* gather list, as in occam_compact */
  const void* src[OCCAM_MAX_GATHER];
  int64_t row_bytes[OCCAM_MAX_GATHER];
  void* dst[OCCAM_MAX_GATHER];
  int64_t capacity_rows;
  /* OCCAM_RULE_REGISTER (0, the method), OCCAM_RULE_MEAN (ref1 and ref2
   * become the mean scores of the segment's visual rows and of the sample's
   * visual S1 rows, as occam_mean_reference computes them; the outputs ref1
   * and ref2 hold those means) or OCCAM_RULE_BUDGET (Stage I unchanged; S2 =
   * occam_budget_keep of s2 over the visual S1 rows with `budget`; lambda2
   * is unused and ref2 keeps the register reference). */
  int32_t rule;
  const int32_t* budget; /* [B] int32 device, OCCAM_RULE_BUDGET only (else unused) */
  /* relative width of the near-threshold band of the optional outputs near1
   * and near2: |s - tau| <= near_rel * |tau|; 0 (or negative, or NaN) means
   * 1e-5, the band inside which a mask may legitimately differ between two
   * correct fp32 evaluations of the scores */
  float near_rel;
} occam_prune_args;

/* Outputs of occam_prune. Required: keep2 [total_rows] u8 (S2, registers =
 * keep_registers), out_index [capacity_rows] int32, count_vis [B] int32
 * (kept visual rows = the sample's budget |S2 \ {r}|), count_out [B] int32,
 * out_off [B+1] int64. Optional (NULL to skip): keep1 [total_rows] u8 (S1,
 * registers = 1), s1 [total_rows], ref1 [S_tot], s2 [total_rows], ref2 [B]
 * (fp32), n1_vis [B] int32 (visual rows of S1), n_eff [S_tot, H1] fp32
 * ([CLS] mode only, else OCCAM_ERR_UNSUPPORTED): per segment and head the
 * effective number of attended keys of the Stage-I [CLS] attention,
 * exp(H(a)) with H(a) = -sum_i a_i log a_i over the keys {[CLS]} u rows
 * (Sec. 3.2, Observation 1). near1, near2 [total_rows] u8 (optional):
 * near-threshold flags of the two tests (Eq. 5 and Eq. 8), the rows whose
 * keep decision turns on the last digits of their score. near1[v] = 1 for a
 * visual row with |s1(v) - tau1| <= near_rel * |tau1| (tau1 = lambda1 * ref1
 * of its segment, the same fp32 product the test uses); near2[v] = 1 for a
 * visual S1 row with |s2(v) - tau2| <= near_rel * |tau2| (tau2 = lambda2 *
 * ref2 of its sample); every other row 0. Under OCCAM_RULE_BUDGET there is
 * no Stage-II threshold and near2 is all 0. */
typedef struct occam_prune_out {
  uint8_t* keep2;
  int32_t* out_index;
  int32_t* count_vis;
  int32_t* count_out;
  int64_t* out_off;
  uint8_t* keep1;
  float* s1;
  float* ref1;
  float* s2;
  float* ref2;
  int32_t* n1_vis;
  float* n_eff;
  uint8_t* near1;
  uint8_t* near2;
} occam_prune_out;

/* The whole path in one call (Algorithm 1's pruning steps): Stage-I scores,
 * S1 (threshold lambda1 per segment), Stage-II scores over S1, S2
 * (threshold lambda2 per sample), compaction and gather. Part of Stage II
 * runs on a second stream that the library owns (one per host thread,
 * device and `stream`, created on first use), forked from and joined back to
 * `stream` with events, so the call stays ordered on `stream` and can be
 * captured into a CUDA graph. Calls on different streams with their own
 * workspaces and outputs may be in flight at once (consecutive batches of a
 * serving loop); their kernels then share the GPU. */
int occam_prune(const occam_prune_args* args, const occam_prune_out* out, void* workspace,
                size_t workspace_bytes, occam_stream_t stream);
/* Memory kinds (occam_prune and occam_prune_traced): q, k_cls, K1, Q_text,
 * K_text and K2 must be device (or managed) memory, since they are read by
 * TMA copies; gather sources and destinations may also be pinned host
 * memory. Anything else returns OCCAM_ERR_INVALID_ARG. */

/* occam_prune for inputs that stay in host memory (a GB300 host's memory is
 * reachable from the GPU). The paper has no counterpart: this is the
 * deployment path for callers whose K2 and gather tensors live on the host.
 * Arguments are those of occam_prune, with two differences:
 *   - args->stage2.K2 and the gather sources args->src[t] (and destinations
 *     args->dst[t]) may be pinned host memory (cudaHostAlloc /
 *     cudaHostRegister); pageable host memory is refused with
 *     OCCAM_ERR_INVALID_ARG. The scoring inputs (q, k_cls, K1, Q_text,
 *     K_text) must be device memory, as for occam_prune.
 *   - k2_stage: device memory of at least total_rows * H2 * d2 * 2 bytes,
 *     16-byte aligned, owned by the caller. After Stage I the call copies
 *     the S1 rows of K2, and only those, into k2_stage at their own row
 *     positions; Stage II then reads k2_stage. Its other rows are left as
 *     they are.
 * A gather source equal to K2 (same pointer, row_bytes = H2 * d2 * 2) is
 * read from k2_stage, since every kept row is an S1 row. So only the S1
 * rows of K2 and the kept rows of the other gather sources cross the host
 * link, not whole tensors. Results are identical to occam_prune on
 * the same values. In occam_prune_traced's event order the copy falls in the
 * interval after the Stage-I finalize. */
int occam_prune_staged(const occam_prune_args* args, const occam_prune_out* out, void* k2_stage,
                       size_t k2_stage_bytes, void* workspace, size_t workspace_bytes, occam_stream_t stream);

/* occam_prune that also records caller-created CUDA events (cudaEvent_t,
 * passed as void*) on `stream` between its steps, for per-kernel timing:
 * events[0] after the initial zeroing, then one after each step in launch
 * order: [CLS] or mutual scoring, Stage-I finalize, S1 list + work plan,
 * fused tensor-core Stage II, two-pass Stage II (statistics and scores
 * kernels, for the samples the fused kernel does not take), compaction scan,
 * gather. Mutual scoring and the two-pass Stage II are two kernels each,
 * timed together. When the fused kernel is enabled the two-pass kernels run
 * on a second stream beside it, so the fused interval covers all of Stage II
 * and the two-pass interval is empty. Extra events are left unrecorded;
 * missing ones are skipped. Results are identical to occam_prune. */
int occam_prune_traced(const occam_prune_args* args, const occam_prune_out* out, void* workspace,
                       size_t workspace_bytes, occam_stream_t stream, void* const* events, int32_t n_events);

/* occam_compact for callers that cannot allocate device memory. The paper
 * has no counterpart: this is a deployment convenience. Some callers may not
 * call cudaMalloc at all -- plugins whose host framework owns every device
 * allocation, serving runtimes that forbid allocation once started, or code
 * that must not grow the device footprint per call -- and so cannot supply
 * the workspace occam_compact needs for its scan state. This entry point
 * takes the same arguments as occam_compact minus the workspace: its scratch
 * (scan tile states, a tile ticket, a status word) is a fixed 64.25 KiB
 * array inside this library, present on every GPU that loads the library
 * until the process exits. It calls no cudaMalloc, cudaFree or allocating
 * library routine. Limits and behaviour:
 * - total_rows <= 16,777,216 (8,192 scan tiles of 2,048 rows); larger batches
 *   are rejected with OCCAM_ERR_UNSUPPORTED and nothing is launched.
 * - The first call in a CUDA context (normally a device's primary context),
 *   made with that device current, looks up the array's device address
 *   (cudaGetSymbolAddress) and caches it under the context's unique id; make
 *   that first call before any stream capture. A context created later on
 *   the same device (after cudaDeviceReset, say) gets a fresh lookup.
 * - Arguments are checked exactly as occam_compact checks them.
 * - All calls on a device share the one array. Each call clears the parts it
 *   needs before use, but calls that overlap on the GPU (different streams
 *   without ordering, or different host threads) race on it and produce
 *   wrong results: order them.
 * - Device-side errors are not reported (there is no workspace status word to
 *   read): a capacity overflow shows as out_off[B] > capacity_rows, with
 *   counts and offsets still exact. The scan's bounded look-back wait, a
 *   guard against a fault that correct operation never reaches, is not
 *   reported either: if it ran out, the outputs would be undefined. */
int occam_compact_noalloc(const occam_batch* batch, const uint8_t* keep, int32_t n_tensors,
                          const void* const* src, const int64_t* row_bytes, void* const* dst,
                          int64_t capacity_rows, int32_t* out_index, int32_t* count_out, int64_t* out_off,
                          occam_stream_t stream);

/* Diagnostic of the bounded device-side waits (no fault, trap or hang). One
 * warp waits, each time for about limit_ns (1 .. 1e9), on an mbarrier that
 * nothing completes (the tensor-core kernels' timer-bounded wait and the
 * streaming kernels' iteration-bounded wait) and on a flag that nothing sets
 * (the look-backs' spin). scratch: 4 int32, device. It is zeroed first; on
 * completion scratch[0] = a bitmask of the waits that gave up (7 when all
 * three did) and scratch[1] = OCCAM_ERR_TIMEOUT if any did, else 0; scratch[2..3] is the
 * flag. The context stays usable afterwards. */
int occam_selftest_wait(uint64_t limit_ns, int32_t* scratch, occam_stream_t stream);

/* How many kernels the last entry point called on this host thread launched
 * (host-side count; an entry point that returned an error may have launched
 * fewer than a full call). A launch whose work list turns out empty on the
 * device still counts. */
int occam_last_call_kernels(void);

/* Library version string (static storage). */
const char* occam_version(void);

/* Stage-II routing, for tests and diagnostics only (the paper has no
 * counterpart). OCCAM_ROUTE_AUTO (the default, and what a deployment uses):
 * each sample takes the fused tensor-core kernel where its S1 fits, small
 * batches on wider clusters; OCCAM_ROUTE_TWOPASS: every sample takes the
 * two-pass kernels; OCCAM_ROUTE_NARROW: AUTO without the wider clusters.
 * Results agree across routes within the scores' tolerance; the switch lets
 * tests reach every path on the same inputs. Process-wide; it applies to
 * calls made after it returns. previous (host, nullable) receives the route
 * in force before the call. An unknown route returns OCCAM_ERR_INVALID_ARG
 * and changes nothing. */
#define OCCAM_ROUTE_AUTO 0
#define OCCAM_ROUTE_TWOPASS 1
#define OCCAM_ROUTE_NARROW 2
int occam_set_stage2_route(int32_t route, int32_t* previous);

#ifdef __cplusplus
}
#endif

#endif /* OCCAM_H */
