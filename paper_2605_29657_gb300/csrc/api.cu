// api.cu -- the C ABI of include/occam.h: host-side validation, workspace
// carve-up and kernel launches. Nothing here allocates memory.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <utility>

#include "common.cuh"
#include "kernels.cuh"
#include "nvtx.cuh"
#include "validate.cuh"

using namespace occam;

int& occam::launch_counter() {
  thread_local int n = 0;
  return n;
}

namespace {

constexpr size_t kAlign = 256;

size_t align_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }


WsLayout ws_layout(const occam_batch* b, int H1, int H2) {
  WsLayout L{};
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = align_up(off + (bytes ? bytes : 1));
    return o;
  };
  const int64_t rows = b->total_rows, S = b->S_tot, B = b->B, T = b->total_text;
  L.status = take(4);
  // accumulators zeroed at the start of every prune call: one contiguous range
  L.zero_begin = off;
  L.counters = take(CNT_SLOTS * 4);
  L.done = take(B * 4);
  L.scan_tiles = cdiv(rows, kScanTile);
  L.scan_state = take(L.scan_tiles * 8);
  L.seg_state = take(S * 8);
  L.zero_end = off;
  L.role = take(rows);
  L.keep1 = take(rows);
  L.s1 = take(rows * 4);
  L.s2 = take(rows * 4);
  L.ref1 = take(S * 4);
  L.dense = take(rows * 4);
  L.n1 = take(B * 4);
  L.n1_vis = take(B * 4);
  const int64_t tps = cdiv(b->max_text, kTextTile);
  const int64_t nhg = cdiv(H2 > 0 ? H2 : 1, kHeadGroup);
  const int64_t chmax = cdiv(b->max_sample_rows, kKeyChunk);
  L.maxA = B * tps * nhg * kStatSplits;
  L.maxB = B * tps * chmax;
  // fused items: one per text tile, or kHsGroups per tile of a head-split batch
  L.maxF = std::max<int64_t>(B * cdiv(b->max_text, 128), kHsMaxTiles * kHsGroups);
  L.maxSlots = L.maxB + L.maxF * kFusedSlotsPerItem16;
  L.itemsF = take(L.maxF * 16);
  L.itemsF8 = take(L.maxF * 16);
  L.itemsF16 = take(L.maxF * 16);
  L.itemsHS = take(kHsMaxTiles * 16);
  // head-split scratch only for batches with at most kHsMaxTiles text tiles
  L.ppart = (B * cdiv(b->max_text, kHsRows) <= kHsMaxTiles)
                ? take((size_t)kHsMaxTiles * kHsGroups * 16 * kHsRows * kFusedMaxOwnImg * 4)
                : 0;
  L.itemA_off = take((B + 1) * 4);
  L.itemB_off = take((B + 1) * 4);
  L.slot_off = take((B + 1) * 4);
  L.stats2 = take(T * (H2 > 0 ? H2 : 1) * kStatSplits * 8);
  L.refpart = take(L.maxSlots * 4);
  L.ref2 = take(B * 4);
  L.tau2 = take(B * 4);
  L.stats1_rows = rows;
  L.stats1 = take(rows * (H1 > 0 ? H1 : 1) * 8);
  L.l2sel = take(kL2SelBytes);
  L.total = off;
  return L;
}

template <typename T>
T* at(void* ws, size_t off) {
  return reinterpret_cast<T*>(static_cast<unsigned char*>(ws) + off);
}

int check_ws(const occam_batch* b, int H1, int H2, void* ws, size_t bytes, WsLayout* L) {
  *L = ws_layout(b, H1, H2);
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & (kAlign - 1)) != 0 || bytes < L->total)
    return OCCAM_ERR_WORKSPACE;
  return OCCAM_OK;
}

BatchDev dev_batch(const occam_batch* b) {
  BatchDev d;
  d.B = b->B;
  d.S_tot = b->S_tot;
  d.total_rows = b->total_rows;
  d.total_text = b->total_text;
  d.row_off = b->row_off;
  d.seg_off = b->seg_off;
  d.seg_first = b->seg_first;
  d.seg_sample = b->seg_sample;
  d.reg_idx = b->reg_idx;
  d.reg_off = b->reg_off;
  d.text_off = b->text_off;
  return d;
}

int num_sms() {
  static int n = 0;
  static std::once_flag once;
  std::call_once(once, [] {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 148;
  });
  return n;
}

// the finalize kernel's shared copy of a segment: s1 (4 B) and role (1 B) per row
size_t finalize_smem_bytes(int rows) { return ((size_t)rows * (4 + 1) + 15) & ~(size_t)15; }

void set_smem_attrs() {
  static std::once_flag once;
  std::call_once(once, [] {
    cudaFuncSetAttribute(stage1_finalize_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)finalize_smem_bytes(kFinalizeSmemRows));
  });
}

// cuTensorMapEncodeTiled from the driver, looked up once.
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
  });
  return fn;
}

// A second stream (and fork / join events) per host thread, device and
// caller stream, made on first use and kept for the life of the thread:
// per-thread so that calls from different host threads never share an event,
// per caller stream so that calls in flight on different streams (a serving
// loop's consecutive batches) do not queue behind each other's second
// stream. Past kMaxEntries caller streams, further ones share one entry per
// device (still correct: the events order every use).
struct SideStream {
  cudaStream_t stream = nullptr;
  cudaEvent_t fork = nullptr, join = nullptr;
  bool ok = false;
};

SideStream& side_stream(cudaStream_t caller) {
  constexpr int kMaxEntries = 16, kMaxDevices = 64;
  struct Entry {
    int dev = -1;
    cudaStream_t caller = nullptr;
    SideStream side;
  };
  thread_local Entry table[kMaxEntries];
  thread_local SideStream overflow[kMaxDevices];
  static SideStream bad;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return bad;
  SideStream* s = nullptr;
  for (Entry& e : table) {
    if (e.dev == dev && e.caller == caller) {
      s = &e.side;
      break;
    }
  }
  if (!s) {
    for (Entry& e : table) {
      if (e.dev < 0) {
        e.dev = dev;
        e.caller = caller;
        s = &e.side;
        break;
      }
    }
  }
  if (!s) s = &overflow[dev];
  if (!s->ok) {
    s->ok = cudaStreamCreateWithFlags(&s->stream, cudaStreamNonBlocking) == cudaSuccess &&
            cudaEventCreateWithFlags(&s->fork, cudaEventDisableTiming) == cudaSuccess &&
            cudaEventCreateWithFlags(&s->join, cudaEventDisableTiming) == cudaSuccess;
  }
  return *s;
}

// Launches kern with the programmatic stream-serialization attribute: it may
// start before the kernel ahead of it in the stream has finished, and waits
// for that kernel's results where it calls pdl_wait() (common.cuh).
template <class... P, class... A>
cudaError_t launch_pdl(void (*kern)(P...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, A&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<A>(args)...);
}

// 2-D bf16 map over a [rows, cols] row-major tensor, 128-byte swizzle, box
// of 64 columns x box_rows rows.
bool encode_map(CUtensorMap* m, const void* base, int64_t rows, int64_t cols, uint32_t box_rows) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  cuuint64_t gdim[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t gstride[1] = {(cuuint64_t)(cols * 2)};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t es[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), gdim, gstride, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D bf16 map over a [rows, heads, dims] tensor, box of box_dims dims x 1
// head x 128 rows: 64 dims with the 128-byte swizzle, or 16 dims with the
// 32-byte swizzle; dims past `dims` read as zero.
bool encode_map3(CUtensorMap* m, const void* base, int64_t rows, int heads, int dims, uint32_t box_dims = 64) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  cuuint64_t gdim[3] = {(cuuint64_t)dims, (cuuint64_t)heads, (cuuint64_t)rows};
  cuuint64_t gstride[2] = {(cuuint64_t)dims * 2, (cuuint64_t)heads * dims * 2};
  cuuint32_t box[3] = {box_dims, 1, 128};
  cuuint32_t es[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), gdim, gstride, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, box_dims == 64 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_32B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Stage-II path selection (occam_set_stage2_route): the fused tensor-core
// kernel for every sample that fits it (AUTO, the default), the two-pass
// kernels for all samples (TWOPASS), or AUTO without widening the clusters of
// small batches (NARROW); the last two let tests reach every path.
std::atomic<int> g_route{OCCAM_ROUTE_AUTO};
bool fused_enabled() { return g_route.load(std::memory_order_relaxed) != OCCAM_ROUTE_TWOPASS; }
bool widening_enabled() { return g_route.load(std::memory_order_relaxed) != OCCAM_ROUTE_NARROW; }

int cuda_ok() {
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? OCCAM_OK : OCCAM_ERR_CUDA;
}

#define OCCAM_TRY(x)                \
  do {                              \
    int _rc = (x);                  \
    if (_rc != OCCAM_OK) return _rc; \
  } while (0)

#define OCCAM_CUDA(x)                                    \
  do {                                                   \
    if ((x) != cudaSuccess) return OCCAM_ERR_CUDA;       \
  } while (0)

int check_stage1(const occam_batch* b, const occam_stage1_args* a) {
  if (!a || !a->q || !a->K1) return OCCAM_ERR_INVALID_ARG;
  if (!aligned16(a->q) || !aligned16(a->K1) || (a->k_cls && !aligned16(a->k_cls))) return OCCAM_ERR_INVALID_ARG;
  if (a->mode == OCCAM_STAGE1_CLS) {
    if (a->H1 != 16 || (a->d1 != 64 && a->d1 != 72 && a->d1 != 128)) return OCCAM_ERR_UNSUPPORTED;
  } else if (a->mode == OCCAM_STAGE1_MUTUAL) {
    if (a->H1 < 1 || a->H1 > 64) return OCCAM_ERR_UNSUPPORTED;
    if (a->d1 != 64 && a->d1 != 72 && a->d1 != 80) return OCCAM_ERR_UNSUPPORTED;
    // work items of the first pass, S_tot * tiles * H1, are int32
    if ((int64_t)b->S_tot * cdiv(b->max_seg_rows, 128) * a->H1 > 0x7fffff00) return OCCAM_ERR_UNSUPPORTED;
  } else {
    return OCCAM_ERR_INVALID_ARG;
  }
  return OCCAM_OK;
}

// Key / value heads of Stage II: H2_kv, where 0 stands for H2.
int kv_heads(const occam_stage2_args* a) { return a->H2_kv > 0 ? a->H2_kv : a->H2; }

int check_stage2(const occam_stage2_args* a) {
  if (!a || !a->Q_text || !a->K2) return OCCAM_ERR_INVALID_ARG;
  if (a->d2 != 128 || a->H2 < 1 || a->H2 > 64) return OCCAM_ERR_UNSUPPORTED;
  if (a->H2_kv < 0 || a->H2 % kv_heads(a) != 0) return OCCAM_ERR_INVALID_ARG;
  if (!aligned16(a->Q_text) || !aligned16(a->K2) || (a->K_text && !aligned16(a->K_text)))
    return OCCAM_ERR_INVALID_ARG;
  return OCCAM_OK;
}

// Memory kinds: the TMA-read inputs must live in device (or managed) memory;
// the K2 of a staged call and gather sources / destinations may also be
// pinned host memory, which kernels reach through its device-side address.
// Pageable (unregistered) host memory is refused: a kernel cannot be sure
// to reach it.
int require_device(const void* p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return OCCAM_ERR_INVALID_ARG;
  }
  return (at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged) ? OCCAM_OK : OCCAM_ERR_INVALID_ARG;
}

int device_view(const void* p, const void** dev) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return OCCAM_ERR_INVALID_ARG;
  }
  if (at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged) {
    *dev = p;
    return OCCAM_OK;
  }
  if (at.type == cudaMemoryTypeHost && at.devicePointer) {
    // the same byte offset into the allocation, seen from the device
    *dev = static_cast<const char*>(at.devicePointer) +
           (static_cast<const char*>(p) - static_cast<const char*>(at.hostPointer));
    return OCCAM_OK;
  }
  return OCCAM_ERR_INVALID_ARG;
}

// Optional CUDA events recorded between the kernels of one call (for live
// per-kernel timing by the caller). mark() records the next event, if any.
struct Trace {
  cudaEvent_t* ev = nullptr;
  int n = 0;
  int* next = nullptr;
  void mark(cudaStream_t st) const {
    if (ev && next && *next < n) cudaEventRecord(ev[(*next)++], st);
  }
};

// ---------------------------------------------------------------- launch helpers

int launch_stage1_scores(const occam_batch* b, const occam_stage1_args* a, const WsLayout& L, void* ws,
                         float* s1, float* s2_zero, cudaStream_t st, Trace trace = Trace()) {
  const NvtxRange nvtx(a->mode == OCCAM_STAGE1_CLS ? "stage1_cls_scores" : "stage1_mutual_scores");
  const BatchDev bt = dev_batch(b);
  int* status = at<int>(ws, L.status);
  if (a->mode == OCCAM_STAGE1_CLS) {
    // per-head logits only; the finalize kernel forms s1 from them
    Stage1ClsParams p;
    p.bt = bt;
    p.q_cls = static_cast<const __nv_bfloat16*>(a->q);
    p.K1 = static_cast<const __nv_bfloat16*>(a->K1);
    p.scale = (float)(1.4426950408889634 / std::sqrt((double)a->d1));  // logits in log2 units
    p.logits = at<float>(ws, L.stats1);
    p.status = status;
    const int64_t tiles = cdiv(b->total_rows, 16);
    const int grid = (int)std::max<int64_t>(1, std::min<int64_t>(tiles, 2 * num_sms()));
    launch_stage1_logits(p, a->d1, grid, st);
    count_launch();
    trace.mark(st);
  } else {
    MutualTcParams p;
    p.bt = bt;
    p.H = a->H1;
    p.d1 = a->d1;
    p.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)a->d1));
    p.inv_h = 1.0f / (float)a->H1;
    p.lsum = at<float>(ws, L.stats1);
    p.s1 = s1;
    p.s2_zero = s2_zero;
    p.status = status;
    // Q1 and K1 as [rows, H1, d1]: boxes of 64 dims x 1 head x 128 rows
    CUtensorMap mq, mk, mq1, mk1;
    if (!encode_map3(&mq, a->q, b->total_rows, a->H1, a->d1) || !encode_map3(&mk, a->K1, b->total_rows, a->H1, a->d1) ||
        !encode_map3(&mq1, a->q, b->total_rows, a->H1, a->d1, 16) ||
        !encode_map3(&mk1, a->K1, b->total_rows, a->H1, a->d1, 16))
      return OCCAM_ERR_CUDA;
    p.tiles = (int)cdiv(b->max_seg_rows, 128);
    p.hgroups = (int)cdiv(a->H1, kMutHeadGroup);
    p.part = p.lsum + (int64_t)a->H1 * b->total_rows;  // stats1 holds 2 * H1 floats per row
    p.queue = at<int32_t>(ws, L.counters) + CNT_MUT;
    OCCAM_CUDA(cudaMemsetAsync(p.queue, 0, 2 * sizeof(int32_t), st));
    launch_mutual_tc(p, mq, mk, mq1, mk1, num_sms(), st);
    trace.mark(st);
  }
  return cuda_ok();
}

// a1 (nullable): in [CLS] mode s1 is formed here from the logits of
// launch_stage1_scores and written to s1; s2_zero (nullable) is zeroed.
// plan (nullable): the last CTA also builds the Stage-II work plan, and
// zeroes the compaction counts count_out / count_vis (nullable).
int launch_finalize1(const occam_batch* b, const WsLayout& L, void* ws, float* s1, const uint8_t* keep_in,
                     float lambda1, int do_threshold, float* ref1, uint8_t* keep1, int32_t* n1_vis,
                     const occam_stage1_args* a1, float* s2_zero, const Stage2Params* plan, int32_t* count_out,
                     int32_t* count_vis, cudaStream_t st, Trace trace = Trace(), float* n_eff = nullptr,
                     int ref_mean = 0, uint8_t* near1 = nullptr, float near_rel = 1e-5f, bool pdl = false) {
  const NvtxRange nvtx("stage1_finalize");
  Stage1FinalizeParams p;
  p.bt = dev_batch(b);
  const bool cls = a1 && a1->mode == OCCAM_STAGE1_CLS;
  p.logits = cls ? at<float>(ws, L.stats1) : nullptr;
  p.q_cls = cls ? static_cast<const __nv_bfloat16*>(a1->q) : nullptr;
  p.k_cls = cls ? static_cast<const __nv_bfloat16*>(a1->k_cls) : nullptr;
  p.scale = cls ? (float)(1.4426950408889634 / std::sqrt((double)a1->d1)) : 1.f;  // log2 units, as the logits
  p.d1 = cls ? a1->d1 : 64;
  p.s1_out = s1;
  p.n_eff = cls ? n_eff : nullptr;
  p.s2_zero = cls ? s2_zero : nullptr;
  // a segment's s1 (4 B/row) and roles (1 B/row) are staged in shared
  // memory when it fits (at most 110 KB)
  p.smem_rows = s1 ? (int)std::min<int64_t>(b->max_seg_rows, kFinalizeSmemRows) : 0;
  p.s1 = s1;
  p.keep_in = keep_in;
  p.lambda1 = lambda1;
  p.ref_mean = ref_mean;
  p.do_threshold = do_threshold;
  p.ref1 = ref1;
  p.role = at<uint8_t>(ws, L.role);
  p.keep1 = keep1;
  p.status = at<int>(ws, L.status);
  p.dense = at<int32_t>(ws, L.dense);
  p.n1 = at<int32_t>(ws, L.n1);
  p.n1_vis = n1_vis;
  p.seg_state = at<unsigned long long>(ws, L.seg_state);
  p.counters = at<int32_t>(ws, L.counters);
  p.do_plan = plan ? 1 : 0;
  if (plan) p.plan = *plan;
  p.zero_count_out = count_out;
  p.zero_count_vis = count_vis;
  p.near1 = near1;
  p.near_rel = near_rel;
  // pdl (the op before this launch is the Stage-I kernel, which started after
  // the call's counters were zeroed): programmatic dependent launch, so that
  // the finalize kernel's input-only prologue (its segment ticket, the batch
  // offsets, the [CLS] key's own logits) overlaps the end of that kernel
  if (pdl)
    OCCAM_CUDA(launch_pdl(stage1_finalize_kernel, dim3((unsigned)b->S_tot), dim3(256),
                          (size_t)finalize_smem_bytes(p.smem_rows), st, p));
  else
    stage1_finalize_kernel<<<b->S_tot, 256, finalize_smem_bytes(p.smem_rows), st>>>(p);
  count_launch();
  trace.mark(st);
  return cuda_ok();
}

// Stage II for the samples the plan routed to the two-pass kernels; both
// loop over their item lists, which may be empty.
int launch_twopass(const Stage2Params& p, const WsLayout& L, int sms, const occam_batch* b,
                   const occam_stage2_args* a, cudaStream_t st) {
  const int gA = (int)std::min<int64_t>(L.maxA, sms);
  const int gB = (int)std::min<int64_t>(L.maxB, sms);
  if (gA <= 0 && gB <= 0) return OCCAM_OK;
  // both passes on the tensor cores: keys copied from K2 (and the text keys)
  // by row with cp.async, the text queries in TMA boxes of 128 rows
  // (statistics) and 64 rows (scores)
  CUtensorMap mq128, mq64;
  if (!encode_map(&mq128, a->Q_text, b->total_text, (int64_t)a->H2 * 128, kStatsTile)) return OCCAM_ERR_CUDA;
  if (!encode_map(&mq64, a->Q_text, b->total_text, (int64_t)a->H2 * 128, kTextTile)) return OCCAM_ERR_CUDA;
  if (gA > 0 && launch_stats_tc(p, mq128, gA, st) != 0) return OCCAM_ERR_CUDA;
  if (gB > 0 && launch_scores_tc(p, mq64, gB, st) != 0) return OCCAM_ERR_CUDA;
  return OCCAM_OK;
}

// Stage-II parameter block (the same for the plan, built by the Stage-I
// finalize kernel, and for the Stage-II kernels).
Stage2Params stage2_params(const occam_batch* b, const occam_stage2_args* a, const WsLayout& L, void* ws, float* s2,
                           float* ref2, float lambda2) {
  Stage2Params p;
  p.bt = dev_batch(b);
  p.H = a->H2;
  p.Hkv = kv_heads(a);
  p.Q = static_cast<const __nv_bfloat16*>(a->Q_text);
  p.Kt = static_cast<const __nv_bfloat16*>(a->K_text);
  p.K = static_cast<const __nv_bfloat16*>(a->K2);
  p.scale = (float)(1.0 / std::sqrt((double)a->d2));
  p.role = at<uint8_t>(ws, L.role);
  p.dense = at<int32_t>(ws, L.dense);
  p.n1 = at<int32_t>(ws, L.n1);
  p.itemA_off = at<int32_t>(ws, L.itemA_off);
  p.itemB_off = at<int32_t>(ws, L.itemB_off);
  p.counters = at<int32_t>(ws, L.counters);
  p.maxA = L.maxA;
  p.maxB = L.maxB;
  p.stats = at<float2>(ws, L.stats2);
  p.s2 = s2;
  p.refpart = at<float>(ws, L.refpart);
  p.done = at<int32_t>(ws, L.done);
  p.ref2 = ref2;
  p.tau2 = at<float>(ws, L.tau2);
  p.lambda2 = lambda2;
  p.status = at<int>(ws, L.status);
  const bool fused = fused_enabled() && L.maxF > 0 && b->total_text > 0;
  p.itemsF = at<int4>(ws, L.itemsF);
  p.itemsF8 = at<int4>(ws, L.itemsF8);
  p.itemsF16 = at<int4>(ws, L.itemsF16);
  p.slot_off = at<int32_t>(ws, L.slot_off);
  p.maxF = L.maxF;
  p.use_fused = fused ? 1 : 0;
  p.res16 = widening_enabled() ? fused_resident_clusters(16) : 0;
  p.itemsHS = at<int4>(ws, L.itemsHS);
  p.has_ppart = L.ppart != 0 ? 1 : 0;
  p.res8 = widening_enabled() ? fused_resident_clusters(8) : 0;
  return p;
}

// Stage II after the Stage-I finalize kernel planned it (same arguments).
// Clusters a fused launch of C-CTA clusters makes: no more than the device
// holds at once (a cluster must fit in one GPC). Launched clusters beyond
// that cannot be placed until resident ones leave, and while they wait, the
// clusters of the launch beside it on the other stream are not placed either
// (measured: the 8-CTA clusters of the Qwen3-VL-shaped batch started only
// when the 16-CTA launch's surplus clusters were placed). Items come from the
// launch's queue, so fewer clusters lose no work.
int fused_launch_clusters(int C, int64_t max_items, int sms) {
  const int res = fused_resident_clusters(C);
  const int64_t cap = res > 0 ? res : sms / C;
  return (int)std::max<int64_t>(1, std::min<int64_t>(max_items, cap));
}

int launch_stage2(const occam_batch* b, const occam_stage2_args* a, const WsLayout& L, void* ws, float* s2,
                  float* ref2, float lambda2, cudaStream_t st, Trace trace = Trace()) {
  const NvtxRange nvtx("stage2_scores");
  const Stage2Params p = stage2_params(b, a, L, ws, s2, ref2, lambda2);
  const bool fused = p.use_fused != 0;
  trace.mark(st);
  const int sms = num_sms();
  if (fused) {
    CUtensorMap mq;
    const int64_t cols = (int64_t)a->H2 * 128;
    const void* kt = a->K_text ? a->K_text : a->Q_text;
    if (!encode_map(&mq, a->Q_text, b->total_text, cols, 128)) return OCCAM_ERR_CUDA;
    // S1 key rows are gathered four at a time (TMA gather4: box one row
    // high); text key rows, which are consecutive, come in boxes of 16 rows
    CUtensorMap mk, mkt;
    // keys: H2_kv heads per row (grouped-query attention), queries H2
    const int64_t cols_kv = (int64_t)kv_heads(a) * 128;
    if (!encode_map(&mk, a->K2, b->total_rows, cols_kv, 1)) return OCCAM_ERR_CUDA;
    if (!encode_map(&mkt, kt, b->total_text, a->K_text ? cols_kv : cols, 16)) return OCCAM_ERR_CUDA;
    Stage2TcParams q;
    q.bt = p.bt;
    q.H = a->H2;
    q.ppart = L.ppart != 0 ? at<float>(ws, L.ppart) : nullptr;
    q.itemsHS = p.itemsHS;
    q.kv_group = a->H2 / kv_heads(a);
    q.K = static_cast<const __nv_bfloat16*>(a->K2);
    q.Kt = static_cast<const __nv_bfloat16*>(kt);
    q.scale_log2 = p.scale * 1.4426950408889634f;
    q.has_text = a->K_text ? 1 : 0;
    q.dense = p.dense;
    q.n1 = p.n1;
    q.role = p.role;
    q.items = p.itemsF;
    q.counters = p.counters;
    q.s2 = s2;
    q.refpart = p.refpart;
    q.slot_off = p.slot_off;
    q.done = p.done;
    q.ref2 = ref2;
    q.tau2 = p.tau2;
    q.lambda2 = lambda2;
    q.status = p.status;
    // The 8-CTA launch runs beside the 4-CTA one on a second stream (fork and
    // join by events), so SMs one of them leaves idle serve the other. Both
    // launch a cluster per SM group; clusters take items from a queue, so
    // clusters that become resident late simply find less work.
    SideStream& side = side_stream(st);
    if (!side.ok) return OCCAM_ERR_CUDA;
    OCCAM_CUDA(cudaEventRecord(side.fork, st));
    OCCAM_CUDA(cudaStreamWaitEvent(side.stream, side.fork, 0));
    // A batch whose every text tile fits as a resident 16-CTA cluster gets
    // the 16-CTA routing for all of its fused samples (the plan's widening;
    // a sample that a 16-CTA cluster cannot hold fits no smaller one): its
    // 8- and 4-CTA launches would have no items, so they are not made.
    const bool only16 = p.res16 > 0 && (int64_t)b->B * cdiv(b->max_text, 128) <= p.res16;
    Stage2TcParams q8 = q;
    q8.items = p.itemsF8;
    q8.queue = p.counters + CNT_QUEUE8;
    const int ncl8 = fused_launch_clusters(8, L.maxF, sms);
    if (!only16 && launch_fused(8, mq, mk, mkt, q8, ncl8, side.stream) != 0) return OCCAM_ERR_CUDA;
    // samples too large for 8 CTAs: 16-CTA clusters, on this stream ahead of
    // the 4-CTA launch. A launch without items returns at once; it also
    // lets the 8-CTA clusters (larger items) take their SMs first, which
    // measured faster than starting the 4-CTA launch first.
    Stage2TcParams q16 = q;
    q16.items = p.itemsF16;
    q16.queue = p.counters + CNT_QUEUE16;
    const int ncl16 = fused_launch_clusters(16, L.maxF, sms);
    if (launch_fused(16, mq, mk, mkt, q16, ncl16, st) != 0) return OCCAM_ERR_CUDA;
    // head-split tiles (small batches) meet right behind the 16-CTA launch
    launch_s2_merge(q16, st);
    // the two-pass kernels (samples the fused kernel cannot hold; often none)
    // follow the 8-CTA launch on the second stream. They are enqueued after
    // the 16-CTA launch: a CTA of theirs takes a whole SM, and enqueued
    // earlier they held every SM before the 16-CTA clusters, which need 16
    // SMs of one GPC, could be placed.
    OCCAM_TRY(launch_twopass(p, L, sms, b, a, side.stream));
    q.queue = p.counters + CNT_QUEUE4;
    const int ncl4 = fused_launch_clusters(4, L.maxF, sms);
    if (!only16 && launch_fused(4, mq, mk, mkt, q, ncl4, st) != 0) return OCCAM_ERR_CUDA;
    OCCAM_CUDA(cudaEventRecord(side.join, side.stream));
    OCCAM_CUDA(cudaStreamWaitEvent(st, side.join, 0));
    OCCAM_CUDA(cudaGetLastError());
    trace.mark(st);
  } else {
    trace.mark(st);
    OCCAM_TRY(launch_twopass(p, L, sms, b, a, st));
  }
  trace.mark(st);
  return cuda_ok();
}

int launch_compact(const occam_batch* b, const WsLayout& L, void* ws, int mode, const uint8_t* keep_in,
                   const uint8_t* keep1, const float* s2, int keep_registers, uint8_t* keep_out, int n_tensors,
                   const void* const* src, const int64_t* row_bytes, void* const* dst, int64_t capacity,
                   int32_t* out_index, int32_t* count_out, int32_t* count_vis, int64_t* out_off,
                   cudaStream_t st, bool do_memsets = true, Trace trace = Trace(), bool use_role = false,
                   uint8_t* near_out = nullptr, float near_rel = 1e-5f) {
  const NvtxRange nvtx(mode == 1 ? "stage2_threshold_compact" : "compact");
  ScanParams p;
  p.bt = dev_batch(b);
  p.mode = mode;
  p.keep_in = keep_in;
  p.role = (mode == 1 || use_role) ? at<uint8_t>(ws, L.role) : nullptr;
  p.keep1 = keep1;
  p.s2 = s2;
  p.tau2 = at<float>(ws, L.tau2);
  p.keep_registers = keep_registers;
  p.keep_out = keep_out;
  p.capacity = capacity;
  p.out_index = out_index;
  p.count_out = count_out;
  p.count_vis = count_vis;
  p.out_off = out_off;
  p.tile_state = at<unsigned long long>(ws, L.scan_state);
  p.ticket = at<int32_t>(ws, L.counters) + CNT_SCAN_TICKET;
  p.ntiles = L.scan_tiles;
  p.status = at<int>(ws, L.status);
  p.near_out = mode == 1 ? near_out : nullptr;
  p.near_rel = near_rel;
  if (do_memsets) {
    OCCAM_CUDA(cudaMemsetAsync(p.tile_state, 0, L.scan_tiles * 8, st));
    OCCAM_CUDA(cudaMemsetAsync(p.ticket, 0, 4, st));
    OCCAM_CUDA(cudaMemsetAsync(count_out, 0, b->B * 4, st));
    if (count_vis) OCCAM_CUDA(cudaMemsetAsync(count_vis, 0, b->B * 4, st));
  }
  // without memsets just before it, the op ahead of the scan is a kernel that
  // started after the call's counters were zeroed: programmatic dependent
  // launch, the ticket and the row offsets read before that kernel finishes,
  // everything else after (pdl_wait)
  if (!do_memsets)
    OCCAM_CUDA(launch_pdl(scan_kernel, dim3((unsigned)L.scan_tiles), dim3(256), 0, st, p));
  else
    scan_kernel<<<(unsigned)L.scan_tiles, 256, 0, st>>>(p);
  count_launch();
  trace.mark(st);
  if (n_tensors > 0) {
    GatherParams g;
    g.n_tensors = n_tensors;
    for (int t = 0; t < OCCAM_MAX_GATHER; ++t) {
      g.src[t] = t < n_tensors ? static_cast<const unsigned char*>(src[t]) : nullptr;
      g.dst[t] = t < n_tensors ? static_cast<unsigned char*>(dst[t]) : nullptr;
      g.row_bytes[t] = t < n_tensors ? row_bytes[t] : 0;
    }
    g.out_index = out_index;
    g.out_off = out_off;
    g.B = b->B;
    g.capacity = capacity;
    g.src_rows = b->total_rows;
    g.status = at<int>(ws, L.status);
    // programmatic dependent launch: scheduled as the scan ends, it waits for
    // the scan's results inside (pdl_wait)
    OCCAM_CUDA(launch_pdl(gather_kernel, dim3((unsigned)(num_sms() * 4)), dim3(256), 0, st, g));
    count_launch();
  }
  trace.mark(st);
  return cuda_ok();
}

int mark_roles(const occam_batch* b, const WsLayout& L, void* ws, cudaStream_t st) {
  uint8_t* role = at<uint8_t>(ws, L.role);
  OCCAM_CUDA(cudaMemsetAsync(role, 0, b->total_rows, st));
  roles_scatter_kernel<<<64, 256, 0, st>>>(dev_batch(b), role);
  count_launch();
  return cuda_ok();
}

}  // namespace

extern "C" {

int occam_last_call_kernels(void) { return launch_counter(); }

int occam_set_stage2_route(int32_t route, int32_t* previous) {
  if (route != OCCAM_ROUTE_AUTO && route != OCCAM_ROUTE_TWOPASS && route != OCCAM_ROUTE_NARROW)
    return OCCAM_ERR_INVALID_ARG;
  const int old = g_route.exchange(route);
  if (previous) *previous = old;
  return OCCAM_OK;
}

const char* occam_version(void) { return "occam-gb300 0.1 (sm_103a)"; }

int occam_workspace_size(const occam_batch* batch, int32_t H1, int32_t H2, size_t* bytes) {
  OCCAM_TRY(check_batch(batch));
  if (!bytes) return OCCAM_ERR_INVALID_ARG;
  *bytes = ws_layout(batch, H1, H2).total;
  return OCCAM_OK;
}

int occam_get_status(void* workspace, int32_t* status, occam_stream_t stream) {
  if (!workspace || !status) return OCCAM_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int32_t v = 0;
  OCCAM_CUDA(cudaMemcpyAsync(&v, workspace, 4, cudaMemcpyDeviceToHost, st));
  // the status word and, after it, the check site of a checked build
  OCCAM_CUDA(cudaMemsetAsync(workspace, 0, 8, st));
  OCCAM_CUDA(cudaStreamSynchronize(st));
  *status = v;
  return OCCAM_OK;
}

int occam_score_stage1(const occam_batch* batch, const occam_stage1_args* args, float* s1, float* ref1,
                       void* workspace, size_t workspace_bytes, occam_stream_t stream) {
  const NvtxRange nvtx("occam_score_stage1");
  launch_counter() = 0;
  OCCAM_TRY(check_batch(batch));
  OCCAM_TRY(check_stage1(batch, args));
  if (!s1) return OCCAM_ERR_INVALID_ARG;
  WsLayout L;
  OCCAM_TRY(check_ws(batch, args->H1, 1, workspace, workspace_bytes, &L));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  set_smem_attrs();
  OCCAM_TRY(launch_stage1_scores(batch, args, L, workspace, s1, nullptr, st));
  OCCAM_TRY(launch_finalize1(batch, L, workspace, s1, nullptr, 0.f, 0, ref1, nullptr, nullptr, args, nullptr, nullptr,
                             nullptr, nullptr, st, Trace(), nullptr, 0, nullptr, 1e-5f, true));
  return OCCAM_OK;
}

int occam_threshold(const occam_batch* batch, const float* s, const float* ref, int32_t ref_scope, float lambda,
                    const uint8_t* prev_keep, int32_t keep_registers, uint8_t* keep, int32_t* count_vis,
                    void* workspace, size_t workspace_bytes, occam_stream_t stream) {
  const NvtxRange nvtx("occam_threshold");
  launch_counter() = 0;
  OCCAM_TRY(check_batch(batch));
  if (!s || !ref || !keep) return OCCAM_ERR_INVALID_ARG;
  if (ref_scope != OCCAM_REF_SEGMENT && ref_scope != OCCAM_REF_SAMPLE) return OCCAM_ERR_INVALID_ARG;
  if (!(lambda == lambda)) return OCCAM_ERR_INVALID_ARG;
  WsLayout L;
  OCCAM_TRY(check_ws(batch, 1, 1, workspace, workspace_bytes, &L));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  OCCAM_TRY(mark_roles(batch, L, workspace, st));
  if (count_vis) OCCAM_CUDA(cudaMemsetAsync(count_vis, 0, batch->B * 4, st));
  ThresholdParams p;
  p.bt = dev_batch(batch);
  p.s = s;
  p.ref = ref;
  p.ref_scope = ref_scope;
  p.lambda = lambda;
  p.prev_keep = prev_keep;
  p.keep_registers = keep_registers;
  p.role = at<uint8_t>(workspace, L.role);
  p.keep = keep;
  p.count_vis = count_vis;
  threshold_kernel<<<(unsigned)cdiv(batch->total_rows, 256), 256, 0, st>>>(p);
  count_launch();
  return cuda_ok();
}

int occam_mean_reference(const occam_batch* batch, const float* s, int32_t ref_scope, const uint8_t* prev_keep,
                         float* ref, void* workspace, size_t workspace_bytes, occam_stream_t stream) {
  const NvtxRange nvtx("occam_mean_reference");
  launch_counter() = 0;
  OCCAM_TRY(check_batch(batch));
  if (!s || !ref) return OCCAM_ERR_INVALID_ARG;
  if (ref_scope != OCCAM_REF_SEGMENT && ref_scope != OCCAM_REF_SAMPLE) return OCCAM_ERR_INVALID_ARG;
  WsLayout L;
  OCCAM_TRY(check_ws(batch, 1, 1, workspace, workspace_bytes, &L));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  OCCAM_TRY(mark_roles(batch, L, workspace, st));
  MeanRefParams p;
  p.bt = dev_batch(batch);
  p.s = s;
  p.role = at<uint8_t>(workspace, L.role);
  p.prev_keep = prev_keep;
  p.scope = ref_scope;
  p.ref = ref;
  p.lambda = 0.f;
  p.tau = nullptr;
  mean_ref_kernel<<<ref_scope == OCCAM_REF_SEGMENT ? batch->S_tot : batch->B, 256, 0, st>>>(p);
  count_launch();
  return cuda_ok();
}

int occam_pool_scores(const float* s_in, int64_t rows_in, int32_t group, int32_t mode, float* s_out,
                      occam_stream_t stream) {
  const NvtxRange nvtx("occam_pool_scores");
  launch_counter() = 0;
  if (!s_in || !s_out || group < 1 || rows_in < 0 || rows_in % group != 0) return OCCAM_ERR_INVALID_ARG;
  if (mode != OCCAM_POOL_SUM && mode != OCCAM_POOL_MEAN && mode != OCCAM_POOL_MAX) return OCCAM_ERR_INVALID_ARG;
  const int64_t rows_out = rows_in / group;
  if (rows_out == 0) return OCCAM_OK;
  OCCAM_TRY(require_device(s_in));
  OCCAM_TRY(require_device(s_out));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const unsigned blocks = (unsigned)std::min<int64_t>(cdiv(rows_out, 256), (int64_t)num_sms() * 8);
  pool_scores_kernel<<<blocks, 256, 0, st>>>(s_in, rows_out, group, mode, s_out);
  count_launch();
  return cuda_ok();
}

int occam_budget_keep(const occam_batch* batch, const float* s, const uint8_t* prev_keep, const int32_t* budget,
                      int32_t keep_registers, uint8_t* keep, int32_t* count_vis, void* workspace,
                      size_t workspace_bytes, occam_stream_t stream) {
  const NvtxRange nvtx("occam_budget_keep");
  launch_counter() = 0;
  OCCAM_TRY(check_batch(batch));
  if (!s || !budget || !keep) return OCCAM_ERR_INVALID_ARG;
  WsLayout L;
  OCCAM_TRY(check_ws(batch, 1, 1, workspace, workspace_bytes, &L));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  OCCAM_TRY(mark_roles(batch, L, workspace, st));
  BudgetParams p;
  p.bt = dev_batch(batch);
  p.s = s;
  p.role = at<uint8_t>(workspace, L.role);
  p.prev_keep = prev_keep;
  p.budget = budget;
  p.keep_registers = keep_registers;
  p.keep = keep;
  p.count_vis = count_vis;
  budget_keep_kernel<<<batch->B, 1024, 0, st>>>(p);
  count_launch();
  return cuda_ok();
}

int occam_score_stage2(const occam_batch* batch, const occam_stage2_args* args, const uint8_t* keep1, float* s2,
                       float* ref2, void* workspace, size_t workspace_bytes, occam_stream_t stream) {
  const NvtxRange nvtx("occam_score_stage2");
  launch_counter() = 0;
  OCCAM_TRY(check_batch(batch));
  OCCAM_TRY(check_stage2(args));
  if (!keep1 || !s2 || !ref2) return OCCAM_ERR_INVALID_ARG;
  WsLayout L;
  OCCAM_TRY(check_ws(batch, 1, args->H2, workspace, workspace_bytes, &L));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  set_smem_attrs();
  OCCAM_TRY(mark_roles(batch, L, workspace, st));
  OCCAM_CUDA(cudaMemsetAsync(at<unsigned char>(workspace, L.zero_begin), 0, L.zero_end - L.zero_begin, st));
  OCCAM_CUDA(cudaMemsetAsync(s2, 0, batch->total_rows * 4, st));
  // S1 lists from the given mask (registers always in S1) and the Stage-II plan
  const Stage2Params plan = stage2_params(batch, args, L, workspace, s2, ref2, 1.0f);
  OCCAM_TRY(launch_finalize1(batch, L, workspace, nullptr, keep1, 0.f, 1, nullptr, nullptr,
                             at<int32_t>(workspace, L.n1_vis), nullptr, nullptr, &plan, nullptr, nullptr, st));
  return launch_stage2(batch, args, L, workspace, s2, ref2, 1.0f, st);
}

int occam_compact(const occam_batch* batch, const uint8_t* keep, int32_t n_tensors, const void* const* src,
                  const int64_t* row_bytes, void* const* dst, int64_t capacity_rows, int32_t* out_index,
                  int32_t* count_out, int64_t* out_off, void* workspace, size_t workspace_bytes,
                  occam_stream_t stream) {
  const NvtxRange nvtx("occam_compact");
  launch_counter() = 0;
  OCCAM_TRY(check_batch(batch));
  if (!keep || !count_out || !out_off || capacity_rows < 0 || (capacity_rows > 0 && !out_index))
    return OCCAM_ERR_INVALID_ARG;
  OCCAM_TRY(check_gather(n_tensors, src, row_bytes, dst));
  WsLayout L;
  OCCAM_TRY(check_ws(batch, 1, 1, workspace, workspace_bytes, &L));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  return launch_compact(batch, L, workspace, 0, keep, nullptr, nullptr, 0, nullptr, n_tensors, src, row_bytes,
                        dst, capacity_rows, out_index, count_out, nullptr, out_off, st);
}

static int prune_impl(const occam_prune_args* args, const occam_prune_out* out, void* workspace,
                      size_t workspace_bytes, occam_stream_t stream, Trace trace, void* k2_stage = nullptr,
                      size_t k2_stage_bytes = 0) {
  launch_counter() = 0;
  if (!args || !out) return OCCAM_ERR_INVALID_ARG;
  const occam_batch* b = &args->batch;
  OCCAM_TRY(check_batch(b));
  OCCAM_TRY(check_stage1(b, &args->stage1));
  OCCAM_TRY(check_stage2(&args->stage2));
  OCCAM_TRY(check_gather(args->n_tensors, args->src, args->row_bytes, args->dst));
  if (!out->keep2 || !out->count_vis || !out->count_out || !out->out_off || args->capacity_rows < 0 ||
      (args->capacity_rows > 0 && !out->out_index))
    return OCCAM_ERR_INVALID_ARG;
  if (!(args->lambda1 == args->lambda1) || !(args->lambda2 == args->lambda2)) return OCCAM_ERR_INVALID_ARG;
  if (args->rule != OCCAM_RULE_REGISTER && args->rule != OCCAM_RULE_MEAN && args->rule != OCCAM_RULE_BUDGET)
    return OCCAM_ERR_INVALID_ARG;
  if (args->rule == OCCAM_RULE_BUDGET) {
    if (!args->budget) return OCCAM_ERR_INVALID_ARG;
    OCCAM_TRY(require_device(args->budget));
  }
  if (out->n_eff && args->stage1.mode != OCCAM_STAGE1_CLS) return OCCAM_ERR_UNSUPPORTED;
  // the near-threshold band of the optional flags (0, negative or NaN: 1e-5)
  const float near_rel = args->near_rel > 0.f ? args->near_rel : 1e-5f;
  WsLayout L;
  OCCAM_TRY(check_ws(b, args->stage1.H1, args->stage2.H2, workspace, workspace_bytes, &L));
  // memory kinds (see device_view)
  OCCAM_TRY(require_device(args->stage1.q));
  OCCAM_TRY(require_device(args->stage1.K1));
  if (args->stage1.mode == OCCAM_STAGE1_CLS && args->stage1.k_cls) OCCAM_TRY(require_device(args->stage1.k_cls));
  OCCAM_TRY(require_device(args->stage2.Q_text));
  if (args->stage2.K_text) OCCAM_TRY(require_device(args->stage2.K_text));
  occam_stage2_args a2 = args->stage2;
  const void* k2_src = nullptr;
  const int64_t k2_row = (int64_t)kv_heads(&a2) * a2.d2 * 2;
  if (k2_stage) {
    if (!aligned16(k2_stage) || k2_stage_bytes < (size_t)(b->total_rows * k2_row)) return OCCAM_ERR_INVALID_ARG;
    OCCAM_TRY(require_device(k2_stage));
    OCCAM_TRY(device_view(a2.K2, &k2_src));
    a2.K2 = k2_stage;
  } else {
    OCCAM_TRY(require_device(a2.K2));
  }
  const void* src[OCCAM_MAX_GATHER];
  void* dst[OCCAM_MAX_GATHER];
  for (int t = 0; t < args->n_tensors; ++t) {
    if (k2_stage && args->src[t] == args->stage2.K2 && args->row_bytes[t] == k2_row) {
      // the kept rows are S1 rows: a gather of K2 itself reads the staged copy
      src[t] = k2_stage;
    } else {
      OCCAM_TRY(device_view(args->src[t], &src[t]));
    }
    const void* d = nullptr;
    OCCAM_TRY(device_view(args->dst[t], &d));
    dst[t] = const_cast<void*>(d);
  }
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  set_smem_attrs();
  void* ws = workspace;
  float* s1 = out->s1 ? out->s1 : at<float>(ws, L.s1);
  float* s2 = out->s2 ? out->s2 : at<float>(ws, L.s2);
  uint8_t* keep1 = out->keep1 ? out->keep1 : at<uint8_t>(ws, L.keep1);
  int32_t* n1_vis = out->n1_vis ? out->n1_vis : at<int32_t>(ws, L.n1_vis);
  float* ref2 = out->ref2 ? out->ref2 : at<float>(ws, L.ref2);
  // every zero-initialised accumulator of the call, up front
  OCCAM_CUDA(cudaMemsetAsync(at<unsigned char>(ws, L.zero_begin), 0, L.zero_end - L.zero_begin, st));
  trace.mark(st);
  OCCAM_TRY(launch_stage1_scores(b, &args->stage1, L, ws, s1, s2, st, trace));
  const Stage2Params plan = stage2_params(b, &a2, L, ws, s2, ref2, args->lambda2);
  OCCAM_TRY(launch_finalize1(b, L, ws, s1, nullptr, args->lambda1, 1, out->ref1, keep1, n1_vis, &args->stage1, s2,
                             &plan, out->count_out, out->count_vis, st, trace, out->n_eff,
                             args->rule == OCCAM_RULE_MEAN ? 1 : 0, out->near1, near_rel, true));
  if (k2_stage) {
    // the S1 rows of K2 (only those) into the device staging tensor
    const NvtxRange nvtx("stage_k2_rows");
    StageRowsParams sp;
    sp.bt = dev_batch(b);
    sp.src = static_cast<const unsigned char*>(k2_src);
    sp.dst = static_cast<unsigned char*>(k2_stage);
    sp.row_bytes = k2_row;
    sp.dense = at<int32_t>(ws, L.dense);
    sp.n1 = at<int32_t>(ws, L.n1);
    sp.status = at<int>(ws, L.status);
    stage_rows_kernel<<<num_sms() * 4, 256, 0, st>>>(sp);
    count_launch();
    OCCAM_CUDA(cudaGetLastError());
  }
  OCCAM_TRY(launch_stage2(b, &a2, L, ws, s2, ref2, args->lambda2, st, trace));
  if (args->rule == OCCAM_RULE_BUDGET) {
    // S2 = the budget[b] visual S1 rows with the largest s2 per sample, then
    // the compaction of that mask
    const NvtxRange nvtx("stage2_budget");
    BudgetParams bp;
    bp.bt = dev_batch(b);
    bp.s = s2;
    bp.role = at<uint8_t>(ws, L.role);
    bp.prev_keep = keep1;
    bp.budget = args->budget;
    bp.keep_registers = args->keep_registers;
    bp.keep = out->keep2;
    bp.count_vis = nullptr;
    budget_keep_kernel<<<b->B, 1024, 0, st>>>(bp);
    count_launch();
    OCCAM_CUDA(cudaGetLastError());
    // no Stage-II threshold under the budget rule: no near-threshold rows
    if (out->near2) OCCAM_CUDA(cudaMemsetAsync(out->near2, 0, b->total_rows, st));
    return launch_compact(b, L, ws, 0, out->keep2, nullptr, nullptr, args->keep_registers, nullptr, args->n_tensors,
                          src, args->row_bytes, dst, args->capacity_rows, out->out_index, out->count_out,
                          out->count_vis, out->out_off, st, false, trace, true);
  }
  if (args->rule == OCCAM_RULE_MEAN) {
    // the sample's reference becomes the mean s2 of its visual S1 rows
    const NvtxRange nvtx("stage2_mean_reference");
    MeanRefParams mp;
    mp.bt = dev_batch(b);
    mp.s = s2;
    mp.role = at<uint8_t>(ws, L.role);
    mp.prev_keep = keep1;
    mp.scope = OCCAM_REF_SAMPLE;
    mp.ref = ref2;
    mp.lambda = args->lambda2;
    mp.tau = at<float>(ws, L.tau2);
    mean_ref_kernel<<<b->B, 256, 0, st>>>(mp);
    count_launch();
    OCCAM_CUDA(cudaGetLastError());
  }
  return launch_compact(b, L, ws, 1, nullptr, keep1, s2, args->keep_registers, out->keep2, args->n_tensors,
                        src, args->row_bytes, dst, args->capacity_rows, out->out_index,
                        out->count_out, out->count_vis, out->out_off, st, false, trace, false, out->near2, near_rel);
}

int occam_prune(const occam_prune_args* args, const occam_prune_out* out, void* workspace,
                size_t workspace_bytes, occam_stream_t stream) {
  const NvtxRange nvtx("occam_prune");
  return prune_impl(args, out, workspace, workspace_bytes, stream, Trace());
}

int occam_construct_registers(const occam_batch* batch, void* h, int64_t channels, const int32_t* k_reg,
                              int32_t n_k, void* workspace, size_t workspace_bytes, occam_stream_t stream) {
  const NvtxRange nvtx("occam_construct_registers");
  launch_counter() = 0;
  OCCAM_TRY(check_batch(batch));
  if (!h || channels <= 0 || n_k < 0 || (n_k > 0 && !k_reg)) return OCCAM_ERR_INVALID_ARG;
  WsLayout L;
  OCCAM_TRY(check_ws(batch, 1, 1, workspace, workspace_bytes, &L));
  OCCAM_TRY(require_device(h));
  if (n_k == 0 || batch->S_tot == 0) return OCCAM_OK;
  OCCAM_TRY(require_device(k_reg));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  OCCAM_TRY(mark_roles(batch, L, workspace, st));
  RegistersParams p;
  p.bt = dev_batch(batch);
  p.h = static_cast<__nv_bfloat16*>(h);
  p.channels = channels;
  p.k_reg = k_reg;
  p.n_k = n_k;
  p.role = at<uint8_t>(workspace, L.role);
  registers_kernel<<<batch->S_tot, 256, 0, st>>>(p);
  count_launch();
  return cuda_ok();
}

int occam_calibrate_lambda2(const occam_batch* batch, const float* s2, const float* ref2, const uint8_t* keep1,
                            int64_t target_count, float* lambda2_out, int32_t* n_candidates, void* workspace,
                            size_t workspace_bytes, occam_stream_t stream) {
  const NvtxRange nvtx("occam_calibrate_lambda2");
  launch_counter() = 0;
  OCCAM_TRY(check_batch(batch));
  if (!s2 || !ref2 || !keep1 || !lambda2_out) return OCCAM_ERR_INVALID_ARG;
  if (batch->total_rows > (int64_t)0x7fffffff) return OCCAM_ERR_UNSUPPORTED;
  WsLayout L;
  OCCAM_TRY(check_ws(batch, 1, 1, workspace, workspace_bytes, &L));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  OCCAM_TRY(mark_roles(batch, L, workspace, st));
  Lambda2Params p;
  p.bt = dev_batch(batch);
  p.s2 = s2;
  p.ref2 = ref2;
  p.keep1 = keep1;
  p.role = at<uint8_t>(workspace, L.role);
  p.target = target_count;
  p.keys = reinterpret_cast<uint32_t*>(at<int32_t>(workspace, L.dense));
  p.sel = at<unsigned char>(workspace, L.l2sel);
  p.lambda2 = lambda2_out;
  p.n_candidates = n_candidates;
  // keys and top-digit histogram, then per digit a one-CTA bucket choice and
  // the next digit's histogram, the window of kept counts, the choice
  OCCAM_CUDA(cudaMemsetAsync(p.sel, 0, kL2SelBytes, st));
  const unsigned grid = (unsigned)std::max<int64_t>(1, std::min<int64_t>(cdiv(batch->total_rows, 256), (int64_t)num_sms() * 4));
  l2_keys_kernel<<<grid, 256, 0, st>>>(p);
  l2_select_kernel<<<1, 1024, 0, st>>>(p, 0);
  l2_hist_kernel<<<grid, 256, 0, st>>>(p, 1);
  l2_select_kernel<<<1, 1024, 0, st>>>(p, 1);
  l2_hist_kernel<<<grid, 256, 0, st>>>(p, 2);
  l2_select_kernel<<<1, 1024, 0, st>>>(p, 2);
  l2_window_kernel<<<grid, 256, 0, st>>>(p);
  l2_finish_kernel<<<1, 1024, 0, st>>>(p);
  count_launch(8);
  return cuda_ok();
}

int occam_prune_staged(const occam_prune_args* args, const occam_prune_out* out, void* k2_stage,
                       size_t k2_stage_bytes, void* workspace, size_t workspace_bytes, occam_stream_t stream) {
  const NvtxRange nvtx("occam_prune_staged");
  if (!k2_stage) return OCCAM_ERR_INVALID_ARG;
  return prune_impl(args, out, workspace, workspace_bytes, stream, Trace(), k2_stage, k2_stage_bytes);
}

int occam_prune_traced(const occam_prune_args* args, const occam_prune_out* out, void* workspace,
                       size_t workspace_bytes, occam_stream_t stream, void* const* events, int32_t n_events) {
  const NvtxRange nvtx("occam_prune_traced");
  if (n_events < 0 || (n_events > 0 && !events)) return OCCAM_ERR_INVALID_ARG;
  int next = 0;
  Trace t;
  t.ev = reinterpret_cast<cudaEvent_t*>(const_cast<void**>(events));
  t.n = n_events;
  t.next = &next;
  return prune_impl(args, out, workspace, workspace_bytes, stream, t);
}

}  // extern "C"
