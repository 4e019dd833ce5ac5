// C ABI of librolekv (declared in include/rolekv.h): argument checks on the
// host, TMA descriptors, workspace layout and the kernel launches.  Nothing
// here allocates device memory or synchronises.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cmath>
#include <cstdarg>
#include <cstdint>
#include <cstdio>
#include <cstring>
#include <mutex>  // std::call_once

#include <nvtx3/nvToolsExt.h>

#include "internal.h"
#include "rolekv.h"

namespace rolekv {

size_t select_smem_bytes(int n_max);

namespace {

thread_local char g_err[512] = "no error";

// Optional per-launch timing events of this thread (rolekv_set_stage_events).
constexpr int kMaxStageEvents = 8;
thread_local cudaEvent_t g_stage_events[kMaxStageEvents];
thread_local int g_num_stage_events = 0;
thread_local int g_stage_cursor = 0;

void stage_begin() { g_stage_cursor = 0; }

// Timeout self-test (rolekv_selftest_score_timeout): when armed, the next
// two-pass SnapKV score on this thread waits at its per-unit meeting point for
// one arrival more than there are chunks, with this limit.
thread_local bool g_timeout_test_armed = false;
thread_local uint64_t g_timeout_test_ns = 0;
// Checked-build self-test: rows the next kv_compact takes off its output extent.
thread_local int64_t g_shrink_rows = 0;

// An NVTX range over one library call, so that a profiler's timeline shows
// each call, and the kernels it launches, under the call's name.
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

// Records the next stage event (if any) after a kernel launch.
void stage_mark(cudaStream_t stream) {
  if (g_stage_cursor < g_num_stage_events) cudaEventRecord(g_stage_events[g_stage_cursor], stream);
  ++g_stage_cursor;
}

int fail(int code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return code;
}

int cuda_fail(cudaError_t e, const char* what) {
  return fail(ROLEKV_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

constexpr int kRowsMax = 256;
constexpr int kTileKeys = 128;

int64_t to_fixed(float x) { return static_cast<int64_t>(std::floor(static_cast<double>(x) * 1e6 + 0.5)); }

size_t align256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

// ---------------------------------------------------------------- batches --

struct BatchInfo {
  int L, b, Hq, Hkv, G, d, n_max;
  int kept_extra;
  bool varlen;
  int64_t T;
  int64_t n_units;
};

int check_batch(const rolekv_batch* bt, BatchInfo* bi) {
  if (bt == nullptr) return fail(ROLEKV_ERR_INVALID_ARG, "batch is NULL");
  if (bt->L < 1 || bt->b < 1 || bt->Hq < 1 || bt->Hkv < 1 || bt->d < 1 || bt->n_max < 0)
    return fail(ROLEKV_ERR_INVALID_ARG, "batch sizes must be positive (L=%d b=%d Hq=%d Hkv=%d d=%d n_max=%d)",
                bt->L, bt->b, bt->Hq, bt->Hkv, bt->d, bt->n_max);
  if (bt->Hq % bt->Hkv != 0)
    return fail(ROLEKV_ERR_INVALID_ARG, "Hq=%d is not a multiple of Hkv=%d", bt->Hq, bt->Hkv);
  if (bt->kept_extra < 0) return fail(ROLEKV_ERR_INVALID_ARG, "kept_extra=%d must be >= 0", bt->kept_extra);
  bi->kept_extra = bt->kept_extra;
  bi->L = bt->L;
  bi->b = bt->b;
  bi->Hq = bt->Hq;
  bi->Hkv = bt->Hkv;
  bi->G = bt->Hq / bt->Hkv;
  bi->d = bt->d;
  bi->n_max = bt->n_max;
  bi->varlen = bt->seqlens_host != nullptr;
  bi->T = 0;
  if (bi->varlen) {
    if (bt->cu_seqlens_dev == nullptr)
      return fail(ROLEKV_ERR_INVALID_ARG, "varlen batch needs cu_seqlens_dev");
    for (int s = 0; s < bt->b; ++s) {
      const int n = bt->seqlens_host[s];
      if (n < 0 || n > bt->n_max)
        return fail(ROLEKV_ERR_INVALID_ARG, "seqlens[%d]=%d outside [0, n_max=%d]", s, n, bt->n_max);
      bi->T += n;
    }
    if (bi->T > INT32_MAX) return fail(ROLEKV_ERR_UNSUPPORTED, "more than 2^31-1 packed tokens");
  } else {
    bi->T = static_cast<int64_t>(bt->b) * bt->n_max;
  }
  bi->n_units = static_cast<int64_t>(bt->L) * bt->b * bt->Hkv;
  if (bi->n_units > INT32_MAX / 512) return fail(ROLEKV_ERR_UNSUPPORTED, "too many units");
  return ROLEKV_OK;
}

// Largest element offset touched by a tensor (exclusive), for the given
// per-axis extents.
int64_t tensor_span(const rolekv_tensor& t, int L, int b, int H, int64_t rows, int d, bool packed) {
  if (packed) return (L - 1) * t.s_layer + (rows - 1) * t.s_tok + (H - 1) * t.s_head + d;
  return (L - 1) * t.s_layer + (b - 1) * t.s_seq + (H - 1) * t.s_head + (rows - 1) * t.s_tok + d;
}

int check_tensor(const char* name, const rolekv_tensor& t, int d, int H, bool packed, bool for_tma) {
  if (t.ptr == nullptr) return fail(ROLEKV_ERR_INVALID_ARG, "%s: NULL pointer", name);
  if (reinterpret_cast<uintptr_t>(t.ptr) % 16 != 0)
    return fail(ROLEKV_ERR_INVALID_ARG, "%s: pointer not 16-byte aligned", name);
  if (t.s_layer < 0 || t.s_seq < 0 || t.s_head < 0 || t.s_tok < d)
    return fail(ROLEKV_ERR_INVALID_ARG, "%s: bad strides", name);
  if (t.s_layer % 8 || t.s_seq % 8 || t.s_head % 8 || t.s_tok % 8)
    return fail(ROLEKV_ERR_INVALID_ARG, "%s: strides must be multiples of 8 elements", name);
  if (for_tma) {
    if (t.s_layer % t.s_tok || (!packed && t.s_seq % t.s_tok))
      return fail(ROLEKV_ERR_INVALID_ARG, "%s: layer/sequence strides must be multiples of the token stride", name);
    if (t.s_head % t.s_tok != 0 && (H - 1) * t.s_head + d > t.s_tok)
      return fail(ROLEKV_ERR_INVALID_ARG, "%s: heads neither whole token rows nor inside one token row", name);
  }
  return ROLEKV_OK;
}

// ------------------------------------------------------------- tensor maps --

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 2-D bf16 map over the token rows of a tensor: x runs over the s_tok elements
// of a token row, y over the rows; boxes of 64 x box_rows with the 128-byte
// swizzle the MMA descriptors expect.
int make_row_map(CUtensorMap* map, const rolekv_tensor& t, int64_t span, int box_rows) {
  auto fn = encode_fn();
  if (fn == nullptr) return fail(ROLEKV_ERR_CUDA, "cuTensorMapEncodeTiled is not available");
  const int64_t rows = (span + t.s_tok - 1) / t.s_tok;
  if (rows >= (int64_t(1) << 31)) return fail(ROLEKV_ERR_UNSUPPORTED, "tensor has too many token rows for TMA");
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(t.s_tok), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(t.s_tok) * 2};
  cuuint32_t box[2] = {64, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(t.ptr), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(ROLEKV_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d)", static_cast<int>(r));
  return ROLEKV_OK;
}

// A map over V's token rows for the decode producer (box: 64 rows x d, no
// swizzle: the consumers read V rows packed), used when the rows are strided.
// Returns false when the layout does not suit a tensor map (the producer then
// copies row by row).
bool make_decode_v_map(CUtensorMap* map, const rolekv_tensor& v, int64_t span, int d) {
  auto fn = encode_fn();
  if (fn == nullptr || v.s_tok == d || v.s_layer % v.s_tok != 0 || v.s_seq % v.s_tok != 0) return false;
  const int64_t rows = (span + v.s_tok - 1) / v.s_tok;
  if (rows >= (int64_t(1) << 31)) return false;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(v.s_tok), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(v.s_tok) * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(d), 64};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(v.ptr), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int num_sms() {
  static int sms = 0;
  if (sms == 0) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
      sms = 148;
  }
  return sms;
}

// ------------------------------------------------------------ score plans --

struct ScorePlan {
  ScoreArgs a;
  size_t off_partials, off_lse, off_prepool, off_work, bytes;
  int grid1, grid2;
  bool fused;
  int32_t n_items;
  int32_t* work;
};

// Key tiles per work item of the fused SnapKV kernel: small enough that a
// chunk's tiles are still in L2 when pass 2 reads them again, large enough to
// amortise the per-unit meeting point.  Eight chunks per unit at most: the
// grid (152 SMs = 19 x 8) deals a unit's chunks to CTAs of the same round.
constexpr int kFusedChunkTiles = 64;
constexpr int kFusedMaxChunks = 8;

int64_t score_elems(const BatchInfo& bi) {
  return bi.varlen ? static_cast<int64_t>(bi.L) * bi.Hkv * bi.T : bi.n_units * bi.n_max;
}

int plan_score(int mode, const BatchInfo& bi, int W, bool need_partials, bool need_prepool,
               ScorePlan* p, bool fused = false) {
  ScoreArgs& a = p->a;
  std::memset(&a, 0, sizeof(a));
  p->fused = fused;
  if (bi.d != 64 && bi.d != 128)
    return fail(ROLEKV_ERR_UNSUPPORTED, "head dim %d (the score kernels take 64 or 128)", bi.d);
  a.L = bi.L;
  a.b = bi.b;
  a.G = bi.G;
  a.Hkv = bi.Hkv;
  a.d = bi.d;
  a.n_max = bi.n_max;
  a.varlen = bi.varlen;
  a.T = bi.T;
  a.mode = mode;
  a.n_units = static_cast<int32_t>(bi.n_units);
  if (mode == kModeSnapKV) {
    if (W < 8 || W % 8 != 0 || W * bi.G > kRowsMax)
      return fail(ROLEKV_ERR_UNSUPPORTED, "window W=%d must be a multiple of 8 with W*G <= 256 (G=%d)", W, bi.G);
    a.W = W;
    a.P = W;
  } else {
    if (bi.G > 8) return fail(ROLEKV_ERR_UNSUPPORTED, "H2O takes G <= 8 query heads per KV head (G=%d)", bi.G);
    a.P = bi.G <= 4 ? 64 : 32;
  }
  a.nrows = bi.G * a.P;
  a.nrows_pad = a.nrows <= 128 ? 128 : 256;
  const int ntiles = (bi.n_max + kTileKeys - 1) / kTileKeys;
  if (mode == kModeSnapKV) {
    if (p->fused) {
      // at most kFusedMaxChunks chunks per unit (they must all be resident at
      // once), of about kFusedChunkTiles tiles when the sequence allows
      int nc = (ntiles + kFusedChunkTiles - 1) / kFusedChunkTiles;
      nc = nc < 1 ? 1 : (nc > kFusedMaxChunks ? kFusedMaxChunks : nc);
      a.chunk_tiles = ntiles > 0 ? (ntiles + nc - 1) / nc : 1;
    } else {
      a.chunk_tiles = ntiles < 64 ? (ntiles > 0 ? ntiles : 1) : 64;
    }
    a.n_chunks = (ntiles + a.chunk_tiles - 1) / a.chunk_tiles;
    if (a.n_chunks < 1) a.n_chunks = 1;
    p->grid1 = a.n_units * a.n_chunks;
    p->grid2 = p->grid1;
    p->n_items = a.n_units * a.n_chunks;
    a.nrb_max = 1;
  } else {
    a.nrb_max = (bi.n_max + a.P - 1) / a.P;
    p->grid1 = a.n_units * a.nrb_max;
    p->grid2 = p->grid1;                          // pass 2 per query block too
    a.n_chunks = 1;                               // (fused: no cross-CTA exchange)
    p->n_items = a.n_units * a.nrb_max;
  }
  size_t off = 256;   // first 256 bytes reserved
  p->off_partials = off;
  if (need_partials) off += align256(static_cast<size_t>(a.n_units) * a.n_chunks * kRowsMax * 8);
  p->off_lse = off;
  if (!(p->fused && mode == kModeH2O))           // the fused H2O keeps its normalisers on chip
    off += align256(static_cast<size_t>(a.n_units) * a.nrb_max * kRowsMax * 4);
  p->off_prepool = off;
  if (need_prepool) off += align256(static_cast<size_t>(score_elems(bi)) * 4);
  p->off_work = off;
  if (p->fused) off += align256((static_cast<size_t>(a.n_units) + 1) * 4);
  p->bytes = off;
  return ROLEKV_OK;
}

void set_strides(ScoreArgs& a, const rolekv_tensor& k, const rolekv_tensor& q) {
  a.k_layer = k.s_layer;
  a.k_seq = k.s_seq;
  a.k_head = k.s_head;
  a.k_tok = k.s_tok;
  a.q_layer = q.s_layer;
  a.q_seq = q.s_seq;
  a.q_head = q.s_head;
  a.q_tok = q.s_tok;
}

int bind_workspace(ScorePlan& p, void* ws, size_t ws_bytes) {
  if (ws == nullptr || ws_bytes < p.bytes)
    return fail(ROLEKV_ERR_WORKSPACE, "workspace of %zu bytes given, %zu needed", ws_bytes, p.bytes);
  if (reinterpret_cast<uintptr_t>(ws) % 256 != 0)
    return fail(ROLEKV_ERR_WORKSPACE, "workspace must be 256-byte aligned");
  uint8_t* base = static_cast<uint8_t*>(ws);
  p.a.partials = reinterpret_cast<float2*>(base + p.off_partials);
  p.a.lse2 = reinterpret_cast<float*>(base + p.off_lse);
  p.a.ext_partials = static_cast<int64_t>((p.off_lse - p.off_partials) / sizeof(float2));
  p.a.ext_lse2 = static_cast<int64_t>((p.off_prepool - p.off_lse) / sizeof(float));
  p.work = p.fused ? reinterpret_cast<int32_t*>(base + p.off_work) : nullptr;
  return ROLEKV_OK;
}

// SnapKV scores: pass 1 + normalisers (or the caller's LSE) + pass 2, the
// pre-pool scores going to `prepool`.
int run_snapkv(const BatchInfo& bi, const int32_t* cu_seqlens, const rolekv_tensor& q_win,
               const rolekv_tensor& k, int W, float scale, const float* lse_win, float* prepool,
               ScorePlan& p, int32_t* status, cudaStream_t stream) {
  ScoreArgs& a = p.a;
  set_strides(a, k, q_win);
  a.c1 = (scale > 0.f ? scale : 1.0f / std::sqrt(static_cast<float>(bi.d))) * 1.4426950408889634f;
  a.prepool = prepool;
  a.ext_scores = score_elems(bi);
  a.ext_lse_win = static_cast<int64_t>(bi.L) * bi.b * bi.Hq * W;
  a.status = status;
  a.cu_seqlens = cu_seqlens;
  CUtensorMap kmap, qmap;
  int rc = make_row_map(&kmap, k,
                        tensor_span(k, bi.L, bi.b, bi.Hkv, bi.varlen ? bi.T : bi.n_max, bi.d, bi.varlen),
                        kTileKeys);
  if (rc) return rc;
  rc = make_row_map(&qmap, q_win, tensor_span(q_win, bi.L, bi.b, bi.Hq, W, bi.d, false), W);
  if (rc) return rc;
  cudaError_t e;
  if (p.fused) {
    // one persistent launch: both passes with the normalisers formed
    // in-kernel, or pass 2 alone after the caller's normalisers are converted
    FusedArgs fa{};
    fa.s = a;
    fa.work = p.work;
    fa.n_items = p.n_items;
    fa.single = lse_win != nullptr;
    fa.wait_ns = kWaitLimitNs;
    if (!fa.single && g_timeout_test_armed) {
      fa.hold = 1;
      fa.wait_ns = g_timeout_test_ns;
      g_timeout_test_armed = false;
    }
    if (fa.single) {
      e = launch_snapkv_lse(a, lse_win, stream);
      if (e != cudaSuccess) return cuda_fail(e, "snapkv normalisers");
    } else {
      e = cudaMemsetAsync(p.work, 0, (static_cast<size_t>(a.n_units) + 1) * 4, stream);
      if (e != cudaSuccess) return cuda_fail(e, "clearing the work counters");
    }
    e = launch_snapkv_fused(bi.d, kmap, qmap, fa, stream);
    if (e != cudaSuccess) return cuda_fail(e, "snapkv fused score");
    stage_mark(stream);
    return ROLEKV_OK;
  }
  if (lse_win == nullptr) {
    e = launch_attn_pass(0, bi.d, kmap, qmap, a, p.grid1, stream);
    if (e != cudaSuccess) return cuda_fail(e, "snapkv pass 1");
    stage_mark(stream);
  }
  e = launch_snapkv_lse(a, lse_win, stream);
  if (e != cudaSuccess) return cuda_fail(e, "snapkv normalisers");
  stage_mark(stream);
  e = launch_attn_pass(1, bi.d, kmap, qmap, a, p.grid2, stream);
  if (e != cudaSuccess) return cuda_fail(e, "snapkv pass 2");
  stage_mark(stream);
  return ROLEKV_OK;
}

void fill_compact(const BatchInfo& bi, const int32_t* cu_seqlens, int64_t budget_fx,
                  const int32_t* seqlens_host, const rolekv_tensor& k, const rolekv_tensor& v,
                  const int32_t* keep_idx, void* k_out, void* v_out, int32_t* status,
                  CompactArgs* a) {
  std::memset(a, 0, sizeof(*a));
  a->L = bi.L;
  a->b = bi.b;
  a->Hkv = bi.Hkv;
  a->d = bi.d;
  a->n_max = bi.n_max;
  a->varlen = bi.varlen;
  a->budget_fx = budget_fx;
  a->kept_extra = bi.kept_extra;
  a->K_dense = static_cast<int32_t>(kept_rows(bi.n_max, budget_fx, bi.kept_extra));
  a->K_max = a->K_dense;
  a->Ktot = 0;
  if (bi.varlen)
    for (int s = 0; s < bi.b; ++s) a->Ktot += kept_rows(seqlens_host[s], budget_fx, bi.kept_extra);
  a->cu_seqlens = cu_seqlens;
  a->n_units = static_cast<int32_t>(bi.n_units);
  a->k = static_cast<const uint16_t*>(k.ptr);
  a->v = static_cast<const uint16_t*>(v.ptr);
  a->k_layer = k.s_layer;
  a->k_seq = k.s_seq;
  a->k_head = k.s_head;
  a->k_tok = k.s_tok;
  a->v_layer = v.s_layer;
  a->v_seq = v.s_seq;
  a->v_head = v.s_head;
  a->v_tok = v.s_tok;
  a->keep_idx = keep_idx;
  a->k_out = static_cast<uint16_t*>(k_out);
  a->v_out = static_cast<uint16_t*>(v_out);
  a->status = status;
  const int64_t rows = bi.varlen ? bi.T : bi.n_max;
  a->ext_k = tensor_span(k, bi.L, bi.b, bi.Hkv, rows, bi.d, bi.varlen);
  a->ext_v = tensor_span(v, bi.L, bi.b, bi.Hkv, rows, bi.d, bi.varlen);
  a->ext_keep = bi.varlen ? static_cast<int64_t>(bi.L) * bi.Hkv * a->Ktot : bi.n_units * a->K_dense;
  a->ext_out_rows = a->ext_keep;
}

int check_compact_args(const BatchInfo& bi, const rolekv_tensor& k, const rolekv_tensor& v,
                       const int32_t* keep_idx, void* k_out, void* v_out) {
  if (bi.d < 8 || bi.d > 256 || (bi.d & (bi.d - 1)) != 0)
    return fail(ROLEKV_ERR_UNSUPPORTED, "kv_compact takes d a power of two in 8..256 (d=%d)", bi.d);
  if (keep_idx == nullptr || k_out == nullptr || v_out == nullptr)
    return fail(ROLEKV_ERR_INVALID_ARG, "keep_idx, k_out and v_out are required");
  if (reinterpret_cast<uintptr_t>(k_out) % 16 || reinterpret_cast<uintptr_t>(v_out) % 16)
    return fail(ROLEKV_ERR_INVALID_ARG, "k_out/v_out must be 16-byte aligned");
  int rc;
  if ((rc = check_tensor("k", k, bi.d, bi.Hkv, bi.varlen, false))) return rc;
  if ((rc = check_tensor("v", v, bi.d, bi.Hkv, bi.varlen, false))) return rc;
  return ROLEKV_OK;
}

// ---------------------------------------------------------- select / compact --

int fill_select(const BatchInfo& bi, const rolekv_batch* bt, const rolekv_select_params* sp,
                SelectArgs* a) {
  std::memset(a, 0, sizeof(*a));
  if (sp == nullptr) return fail(ROLEKV_ERR_INVALID_ARG, "select params are NULL");
  if (sp->n_roles < 1 || sp->n_roles > ROLEKV_MAX_ROLES)
    return fail(ROLEKV_ERR_UNSUPPORTED, "n_roles=%d outside 1..%d", sp->n_roles, ROLEKV_MAX_ROLES);
  if (!(sp->budget > 0.f) || sp->budget > 1.f)
    return fail(ROLEKV_ERR_INVALID_ARG, "budget %g outside (0, 1]", static_cast<double>(sp->budget));
  if (sp->policy != ROLEKV_POLICY_ROLE_QUOTA && sp->policy != ROLEKV_POLICY_GLOBAL &&
      sp->policy != ROLEKV_POLICY_FAIR && sp->policy != ROLEKV_POLICY_SLACK &&
      sp->policy != ROLEKV_POLICY_CEIL)
    return fail(ROLEKV_ERR_INVALID_ARG, "unknown policy %d", sp->policy);
  if (sp->keep_last < 0) return fail(ROLEKV_ERR_INVALID_ARG, "keep_last=%d must be >= 0", sp->keep_last);
  if (sp->key_role >= sp->n_roles) return fail(ROLEKV_ERR_INVALID_ARG, "key_role %d >= n_roles", sp->key_role);
  if (bi.n_max > ROLEKV_SELECT_MAX_N)
    return fail(ROLEKV_ERR_UNSUPPORTED, "n_max=%d exceeds the %d tokens the selector holds", bi.n_max,
                ROLEKV_SELECT_MAX_N);
  a->L = bi.L;
  a->b = bi.b;
  a->Hkv = bi.Hkv;
  a->n_max = bi.n_max;
  a->varlen = bi.varlen;
  a->T = bi.T;
  a->cu_seqlens = bt->cu_seqlens_dev;
  a->n_units = static_cast<int32_t>(bi.n_units);
  a->n_roles = sp->n_roles;
  a->budget_fx = to_fixed(sp->budget);
  a->policy = sp->policy;
  a->ban_mask = sp->ban_mask;
  a->keep_last = sp->keep_last;
  for (int r = 0; r < ROLEKV_MAX_ROLES; ++r) {
    float al = r < sp->n_roles ? sp->alpha[r] : 0.f;
    if (r == sp->key_role) al = sp->alpha_key;
    if (!(al >= 0.f) || !std::isfinite(al))
      return fail(ROLEKV_ERR_INVALID_ARG, "alpha[%d]=%g must be finite and >= 0", r, static_cast<double>(al));
    a->alpha_fx[r] = ((sp->ban_mask >> r) & 1u) ? 0 : to_fixed(al);
  }
  if (sp->policy == ROLEKV_POLICY_CEIL) {
    // the ceilings of the unsaturated buckets' shares overshoot the budget by
    // less than one slot each, and at least one bucket takes a whole share
    int weighted = 0;
    for (int r = 0; r < sp->n_roles; ++r) weighted += a->alpha_fx[r] > 0;
    if (bi.kept_extra < weighted - 1)
      return fail(ROLEKV_ERR_INVALID_ARG,
                  "the ceiling policy over %d weighted roles needs batch kept_extra >= %d (got %d)",
                  weighted, weighted - 1, bi.kept_extra);
  }
  a->kept_extra = bi.kept_extra;
  a->K_dense = static_cast<int32_t>(kept_rows(bi.n_max, a->budget_fx, bi.kept_extra));
  a->Ktot = 0;
  if (bi.varlen)
    for (int s = 0; s < bi.b; ++s) a->Ktot += kept_rows(bt->seqlens_host[s], a->budget_fx, bi.kept_extra);
  a->ext_scores = score_elems(bi);
  a->ext_roles = bi.varlen ? bi.T : static_cast<int64_t>(bi.b) * bi.n_max;
  a->ext_keep = bi.varlen ? static_cast<int64_t>(bi.L) * bi.Hkv * a->Ktot : bi.n_units * a->K_dense;
  return ROLEKV_OK;
}

}  // namespace
}  // namespace rolekv

// ---------------------------------------------------- no-allocation variant --
//
// Scratch of snapkv_score_noalloc: the pass-1 partial row statistics and the
// per-row normalisers, held in one file-scope device array so that callers who
// cannot allocate device memory (see rolekv.h) still get the two-pass score.
// Every GPU that loads this library reserves the array until the process exits.
static constexpr size_t kNoAllocScratchBytes = size_t(64) << 20;
static __device__ __align__(256) unsigned char rolekv_noalloc_scratch[kNoAllocScratchBytes];

namespace rolekv {
namespace {

// Device address of the scratch array in the current context.  The host-side
// name of the array is only a stand-in; the address is looked up on every
// call (a cheap runtime query), so a context that was reset and made again
// never sees an address from the old one.
int noalloc_scratch(void** out) {
  void* ptr = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&ptr, rolekv_noalloc_scratch);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(scratch)");
  *out = ptr;
  return ROLEKV_OK;
}

}  // namespace
}  // namespace rolekv

using namespace rolekv;

extern "C" {

int64_t rolekv_kept_count(int64_t n, float budget) {
  if (n < 0 || !(budget > 0.f) || budget > 1.f) return -1;
  return kept_slots(n, to_fixed(budget));
}

int64_t rolekv_kept_rows(int64_t n, float budget, int32_t kept_extra) {
  if (n < 0 || kept_extra < 0 || !(budget > 0.f) || budget > 1.f) return -1;
  return kept_rows(n, to_fixed(budget), kept_extra);
}

const char* rolekv_last_error(void) { return g_err; }

const char* rolekv_version(void) { return "rolekv 0.2 (sm_103a)"; }

int rolekv_selftest_wait(int64_t limit_ns, int32_t* status_dev, void* stream) {
  if (status_dev == nullptr) return fail(ROLEKV_ERR_INVALID_ARG, "status_dev is NULL");
  if (limit_ns < 0 || limit_ns > 10000000000LL)
    return fail(ROLEKV_ERR_INVALID_ARG, "limit_ns=%lld outside 0..1e10", static_cast<long long>(limit_ns));
  cudaError_t e = launch_selftest_wait(static_cast<uint64_t>(limit_ns), status_dev,
                                       static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "rolekv_selftest_wait");
  return ROLEKV_OK;
}

int rolekv_workspace_size(int op, const rolekv_batch* batch, int32_t W, size_t* bytes) {
  if (bytes == nullptr) return fail(ROLEKV_ERR_INVALID_ARG, "bytes is NULL");
  BatchInfo bi;
  int rc = check_batch(batch, &bi);
  if (rc) return rc;
  ScorePlan p;
  switch (op) {
    case 0: rc = plan_score(kModeSnapKV, bi, W, true, true, &p, true); break;
    case 1: rc = plan_score(kModeH2O, bi, 0, false, false, &p, true); break;
    case 2: rc = plan_score(kModeSnapKV, bi, W, true, true, &p, true); break;
    default: return fail(ROLEKV_ERR_INVALID_ARG, "unknown op %d", op);
  }
  if (rc) return rc;
  *bytes = p.bytes;
  return ROLEKV_OK;
}

int snapkv_score(const rolekv_batch* batch, rolekv_tensor q_win, rolekv_tensor k, int32_t W,
                 int32_t pool_k, float scale, const float* lse_win, float* scores,
                 float* scores_prepool, void* workspace, size_t workspace_bytes,
                 int32_t* status_dev, void* stream) {
  NvtxRange nvtx("rolekv:snapkv_score");
  BatchInfo bi;
  int rc = check_batch(batch, &bi);
  if (rc) return rc;
  if (pool_k < 1 || pool_k > 15 || pool_k % 2 == 0)
    return fail(ROLEKV_ERR_UNSUPPORTED, "pool_k=%d must be odd, 1..15", pool_k);
  ScorePlan p;
  rc = plan_score(kModeSnapKV, bi, W, lse_win == nullptr, scores_prepool == nullptr, &p, true);
  if (rc) return rc;
  if (bi.T == 0) return ROLEKV_OK;                 // no tokens: nothing to score
  if (scores == nullptr) return fail(ROLEKV_ERR_INVALID_ARG, "scores is NULL");
  if ((rc = check_tensor("q_win", q_win, bi.d, bi.Hq, false, true))) return rc;
  if ((rc = check_tensor("k", k, bi.d, bi.Hkv, bi.varlen, true))) return rc;
  if ((rc = bind_workspace(p, workspace, workspace_bytes))) return rc;
  if (bi.n_max == 0) return ROLEKV_OK;
  // Without pooling, pass 2 writes the scores directly.
  float* pre = scores_prepool ? scores_prepool
               : pool_k == 1  ? scores
                              : reinterpret_cast<float*>(static_cast<uint8_t*>(workspace) + p.off_prepool);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  stage_begin();
  rc = run_snapkv(bi, batch->cu_seqlens_dev, q_win, k, W, scale, lse_win, pre, p, status_dev, st);
  if (rc) return rc;
  const ScoreArgs& a = p.a;
  if (pre == scores) return ROLEKV_OK;
  cudaError_t e = launch_maxpool(a, pre, scores, pool_k, st);
  if (e != cudaSuccess) return cuda_fail(e, "max-pool");
  stage_mark(st);
  return ROLEKV_OK;
}

int h2o_score(const rolekv_batch* batch, rolekv_tensor q, rolekv_tensor k, float scale,
              const float* lse, float* scores, void* workspace, size_t workspace_bytes,
              int32_t* status_dev, void* stream) {
  NvtxRange nvtx("rolekv:h2o_score");
  BatchInfo bi;
  int rc = check_batch(batch, &bi);
  if (rc) return rc;
  ScorePlan p;
  rc = plan_score(kModeH2O, bi, 0, false, false, &p, true);
  if (rc) return rc;
  if (bi.T == 0) return ROLEKV_OK;                 // no tokens: nothing to score
  if (scores == nullptr) return fail(ROLEKV_ERR_INVALID_ARG, "scores is NULL");
  if (reinterpret_cast<uintptr_t>(lse) & 3u) return fail(ROLEKV_ERR_INVALID_ARG, "lse must be 4-byte aligned");
  if ((rc = check_tensor("q", q, bi.d, bi.Hq, bi.varlen, true))) return rc;
  if ((rc = check_tensor("k", k, bi.d, bi.Hkv, bi.varlen, true))) return rc;
  if ((rc = bind_workspace(p, workspace, workspace_bytes))) return rc;
  if (bi.n_max == 0) return ROLEKV_OK;
  ScoreArgs& a = p.a;
  set_strides(a, k, q);
  a.cu_seqlens = batch->cu_seqlens_dev;
  a.c1 = (scale > 0.f ? scale : 1.0f / std::sqrt(static_cast<float>(bi.d))) * 1.4426950408889634f;
  a.prepool = scores;
  a.status = status_dev;
  a.ext_scores = score_elems(bi);
  CUtensorMap kmap, qmap;
  const int64_t rows = bi.varlen ? bi.T : bi.n_max;
  rc = make_row_map(&kmap, k, tensor_span(k, bi.L, bi.b, bi.Hkv, rows, bi.d, bi.varlen), kTileKeys);
  if (rc) return rc;
  rc = make_row_map(&qmap, q, tensor_span(q, bi.L, bi.b, bi.Hq, rows, bi.d, bi.varlen), a.P);
  if (rc) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  stage_begin();
  // every query block adds its column sums into the zeroed scores
  cudaError_t e = cudaMemsetAsync(scores, 0, static_cast<size_t>(score_elems(bi)) * sizeof(float), st);
  if (e != cudaSuccess) return cuda_fail(e, "clearing the scores");
  // one persistent launch: per query block, its row normalisers (pass 1, or
  // the caller's LSE) then its share of the column sums (pass 2)
  FusedArgs fa{};
  fa.s = a;
  fa.work = p.work;
  fa.n_items = p.n_items;
  fa.single = lse != nullptr;
  fa.h2o_lse = lse;
  fa.ext_h2o_lse = static_cast<int64_t>(bi.L) * bi.Hq * (bi.varlen ? bi.T : static_cast<int64_t>(bi.b) * bi.n_max);
  fa.wait_ns = kWaitLimitNs;
  e = launch_snapkv_fused(bi.d, kmap, qmap, fa, st);
  if (e != cudaSuccess) return cuda_fail(e, "h2o fused score");
  stage_mark(st);
  return ROLEKV_OK;
}

int quest_score(const rolekv_batch* batch, rolekv_tensor q_win, rolekv_tensor k, int32_t W,
                int32_t page, float* scores, void* stream) {
  NvtxRange nvtx("rolekv:quest_score");
  BatchInfo bi;
  int rc = check_batch(batch, &bi);
  if (rc) return rc;
  if (bi.d != 64 && bi.d != 128)
    return fail(ROLEKV_ERR_UNSUPPORTED, "head dim %d (quest_score takes 64 or 128)", bi.d);
  if (W < 1) return fail(ROLEKV_ERR_INVALID_ARG, "window W=%d must be >= 1", W);
  if (page < 1 || page > 4096) return fail(ROLEKV_ERR_INVALID_ARG, "page=%d outside 1..4096", page);
  if (bi.T == 0) return ROLEKV_OK;                 // no tokens: nothing to score
  if (scores == nullptr || (reinterpret_cast<uintptr_t>(scores) & 3u))
    return fail(ROLEKV_ERR_INVALID_ARG, "scores must be a non-NULL, 4-byte aligned pointer");
  if ((rc = check_tensor("q_win", q_win, bi.d, bi.Hq, false, false))) return rc;
  if ((rc = check_tensor("k", k, bi.d, bi.Hkv, bi.varlen, false))) return rc;
  if (bi.n_max == 0) return ROLEKV_OK;
  QuestArgs a;
  std::memset(&a, 0, sizeof(a));
  a.L = bi.L;
  a.b = bi.b;
  a.G = bi.G;
  a.Hkv = bi.Hkv;
  a.d = bi.d;
  a.n_max = bi.n_max;
  a.varlen = bi.varlen;
  a.T = bi.T;
  a.cu_seqlens = batch->cu_seqlens_dev;
  a.n_units = static_cast<int32_t>(bi.n_units);
  a.W = W;
  a.page = page;
  a.q = static_cast<const uint16_t*>(q_win.ptr);
  a.q_layer = q_win.s_layer;
  a.q_seq = q_win.s_seq;
  a.q_head = q_win.s_head;
  a.q_tok = q_win.s_tok;
  a.k = static_cast<const uint16_t*>(k.ptr);
  a.k_layer = k.s_layer;
  a.k_seq = k.s_seq;
  a.k_head = k.s_head;
  a.k_tok = k.s_tok;
  a.scores = scores;
  a.ext_scores = score_elems(bi);
  a.ext_q = tensor_span(q_win, bi.L, bi.b, bi.Hq, W, bi.d, false);
  a.ext_k = tensor_span(k, bi.L, bi.b, bi.Hkv, bi.varlen ? bi.T : bi.n_max, bi.d, bi.varlen);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  stage_begin();
  cudaError_t e = launch_quest(a, st);
  if (e != cudaSuccess) return cuda_fail(e, "quest_score");
  stage_mark(st);
  return ROLEKV_OK;
}

int role_alloc_select(const rolekv_batch* batch, const float* scores, const uint8_t* roles,
                      const rolekv_select_params* params, int32_t pool_k, int32_t* keep_idx,
                      uint8_t* keep_mask, int32_t* kept_per_role, int32_t* status_dev,
                      void* stream) {
  NvtxRange nvtx("rolekv:role_alloc_select");
  BatchInfo bi;
  int rc = check_batch(batch, &bi);
  if (rc) return rc;
  if (bi.T > 0 && (scores == nullptr || roles == nullptr || keep_idx == nullptr))
    return fail(ROLEKV_ERR_INVALID_ARG, "scores, roles and keep_idx are required");
  if ((reinterpret_cast<uintptr_t>(scores) & 3u) || (reinterpret_cast<uintptr_t>(keep_idx) & 3u))
    return fail(ROLEKV_ERR_INVALID_ARG, "scores and keep_idx must be 4-byte aligned");
  if (pool_k < 1 || pool_k > 15 || pool_k % 2 == 0)
    return fail(ROLEKV_ERR_UNSUPPORTED, "pool_k=%d must be odd, 1..15", pool_k);
  SelectArgs a;
  if ((rc = fill_select(bi, batch, params, &a))) return rc;
  a.scores = scores;
  a.roles = roles;
  a.pool_k = pool_k;
  a.keep_idx = keep_idx;
  a.keep_mask = keep_mask;
  a.kept_per_role = kept_per_role;
  a.status = status_dev;
  // (a batch without tokens still writes its zero per-role counts)
  stage_begin();
  cudaError_t e = launch_select(a, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "role_alloc_select");
  stage_mark(static_cast<cudaStream_t>(stream));
  return ROLEKV_OK;
}

namespace {
constexpr int kDecodeRowsPerSplit = 1024;

// Splits of at most kDecodeRowsPerSplit rows, equal in length and a multiple
// of the kernel's 64-row stage, so that a unit's splits finish together.
void decode_split(int64_t m_max, int32_t* rows_per_split, int32_t* n_splits) {
  const int64_t ns = m_max > 0 ? (m_max + kDecodeRowsPerSplit - 1) / kDecodeRowsPerSplit : 1;
  int64_t r = (m_max + ns - 1) / ns;
  r = r > 0 ? (r + 63) / 64 * 64 : 64;
  *rows_per_split = static_cast<int32_t>(r);
  *n_splits = static_cast<int32_t>((m_max + r - 1) / r);
}

// Rows of the largest sequence and the packed row total at this budget.
void decode_rows(const BatchInfo& bi, const rolekv_batch* bt, int64_t bfx, int64_t* m_max,
                 int64_t* total) {
  *m_max = 0;
  *total = 0;
  if (bi.varlen) {
    for (int s = 0; s < bi.b; ++s) {
      const int64_t m = kept_rows(bt->seqlens_host[s], bfx, bi.kept_extra);
      *m_max = m > *m_max ? m : *m_max;
      *total += m;
    }
  } else {
    *m_max = kept_rows(bi.n_max, bfx, bi.kept_extra);
    *total = *m_max * bi.b;
  }
}

size_t decode_ws_bytes(const BatchInfo& bi, int64_t m_max) {
  int32_t rps, splits;
  decode_split(m_max, &rps, &splits);
  return static_cast<size_t>(bi.n_units) * static_cast<size_t>(splits > 0 ? splits : 1) * bi.G *
         (bi.d + 2) * sizeof(float);
}
}  // namespace

int rolekv_decode_workspace_size(const rolekv_batch* batch, float budget, size_t* bytes) {
  BatchInfo bi;
  int rc = check_batch(batch, &bi);
  if (rc) return rc;
  if (bytes == nullptr) return fail(ROLEKV_ERR_INVALID_ARG, "bytes is NULL");
  if (!(budget > 0.f) || budget > 1.f)
    return fail(ROLEKV_ERR_INVALID_ARG, "budget %g outside (0, 1]", static_cast<double>(budget));
  int64_t m_max, total;
  decode_rows(bi, batch, to_fixed(budget), &m_max, &total);
  *bytes = decode_ws_bytes(bi, m_max);
  return ROLEKV_OK;
}

int decode_attention(const rolekv_batch* batch, rolekv_tensor q, rolekv_tensor k_cache,
                     rolekv_tensor v_cache, const int32_t* keep_idx, float budget, float scale,
                     float* out, void* workspace, size_t workspace_bytes, int32_t* status_dev,
                     void* stream) {
  NvtxRange nvtx("rolekv:decode_attention");
  BatchInfo bi;
  int rc = check_batch(batch, &bi);
  if (rc) return rc;
  if (bi.d != 64 && bi.d != 128)
    return fail(ROLEKV_ERR_UNSUPPORTED, "head dim %d (decode_attention takes 64 or 128)", bi.d);
  if (bi.G > 8) return fail(ROLEKV_ERR_UNSUPPORTED, "G=%d query heads per KV head (at most 8)", bi.G);
  if (!(budget > 0.f) || budget > 1.f)
    return fail(ROLEKV_ERR_INVALID_ARG, "budget %g outside (0, 1]", static_cast<double>(budget));
  if (out == nullptr || (reinterpret_cast<uintptr_t>(out) & 15u))
    return fail(ROLEKV_ERR_INVALID_ARG, "out must be a non-NULL, 16-byte aligned pointer");
  if (q.ptr == nullptr || (reinterpret_cast<uintptr_t>(q.ptr) & 15u) || q.s_head < bi.d ||
      q.s_layer < 0 || q.s_seq < 0 || (q.s_head % 8) || (q.s_seq % 8) || (q.s_layer % 8))
    return fail(ROLEKV_ERR_INVALID_ARG, "q: NULL, misaligned or bad strides");
  const int64_t bfx = to_fixed(budget);
  int64_t m_max, total;
  decode_rows(bi, batch, bfx, &m_max, &total);
  if (total > 0) {                                 // (no rows: the outputs are zeros)
    if ((rc = check_tensor("k_cache", k_cache, bi.d, bi.Hkv, bi.varlen, false))) return rc;
    if ((rc = check_tensor("v_cache", v_cache, bi.d, bi.Hkv, bi.varlen, false))) return rc;
  }
  const size_t need = decode_ws_bytes(bi, m_max);
  if (workspace == nullptr || workspace_bytes < need)
    return fail(ROLEKV_ERR_WORKSPACE, "workspace of %zu bytes, %zu needed", workspace_bytes, need);
  if (reinterpret_cast<uintptr_t>(workspace) & 255u)
    return fail(ROLEKV_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
  DecodeArgs a;
  std::memset(&a, 0, sizeof(a));
  a.L = bi.L;
  a.b = bi.b;
  a.G = bi.G;
  a.Hkv = bi.Hkv;
  a.d = bi.d;
  a.n_max = bi.n_max;
  a.varlen = bi.varlen;
  a.cu_seqlens = batch->cu_seqlens_dev;
  a.n_units = static_cast<int32_t>(bi.n_units);
  a.budget_fx = bfx;
  a.kept_extra = bi.kept_extra;
  a.Ktot = bi.varlen ? total : 0;
  a.K_dense = bi.varlen ? 0 : static_cast<int32_t>(m_max);
  a.q = static_cast<const uint16_t*>(q.ptr);
  a.q_layer = q.s_layer;
  a.q_seq = q.s_seq;
  a.q_head = q.s_head;
  a.k = static_cast<const uint16_t*>(k_cache.ptr);
  a.k_layer = k_cache.s_layer;
  a.k_seq = k_cache.s_seq;
  a.k_head = k_cache.s_head;
  a.k_tok = k_cache.s_tok;
  a.v = static_cast<const uint16_t*>(v_cache.ptr);
  a.v_layer = v_cache.s_layer;
  a.v_seq = v_cache.s_seq;
  a.v_head = v_cache.s_head;
  a.v_tok = v_cache.s_tok;
  a.keep_idx = keep_idx;
  a.c1 = (scale > 0.f ? scale : 1.0f / std::sqrt(static_cast<float>(bi.d))) * 1.4426950408889634f;
  decode_split(m_max, &a.rows_per_split, &a.n_splits);
  a.part = static_cast<float*>(workspace);
  a.out = out;
  a.o_seq = static_cast<int64_t>(bi.Hq) * bi.d;
  a.o_layer = a.o_seq * bi.b;
  a.o_head = bi.d;
  a.status = status_dev;
  {
    const int64_t rows = bi.varlen ? total : m_max;   // cache rows per (layer, head) / unit
    a.ext_q = tensor_span(q, bi.L, bi.b, bi.Hq, 1, bi.d, false);
    a.ext_k = tensor_span(k_cache, bi.L, bi.b, bi.Hkv, rows, bi.d, bi.varlen);
    a.ext_v = tensor_span(v_cache, bi.L, bi.b, bi.Hkv, rows, bi.d, bi.varlen);
    a.ext_keep = keep_idx == nullptr ? 0 : static_cast<int64_t>(bi.L) * bi.Hkv * (bi.varlen ? total : bi.b * m_max);
    a.ext_part = static_cast<int64_t>(workspace_bytes / sizeof(float));
    a.ext_out = static_cast<int64_t>(bi.L) * bi.b * bi.Hq * bi.d;
  }
  CUtensorMap kmap, vmap;
  std::memset(&kmap, 0, sizeof(kmap));
  std::memset(&vmap, 0, sizeof(vmap));
  if (total > 0) {
    const int64_t rows = bi.varlen ? total : m_max;
    a.v_tma = make_decode_v_map(&vmap, v_cache, tensor_span(v_cache, bi.L, bi.b, bi.Hkv, rows, bi.d, bi.varlen),
                                bi.d) ? 1 : 0;
    // K through a tensor map when its layout suits one (else row by row)
    const bool k_ok = k_cache.s_layer % k_cache.s_tok == 0 && (bi.varlen || k_cache.s_seq % k_cache.s_tok == 0);
    if (k_ok && make_row_map(&kmap, k_cache, tensor_span(k_cache, bi.L, bi.b, bi.Hkv, rows, bi.d, bi.varlen), 64) ==
                    ROLEKV_OK)
      a.k_tma = 1;                                 // (on failure, row-by-row copies)
  }
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  stage_begin();
  cudaError_t e = launch_decode(a, kmap, vmap, st);
  if (e != cudaSuccess) return cuda_fail(e, "decode_attention");
  stage_mark(st);
  return ROLEKV_OK;
}

int kv_compact(const rolekv_batch* batch, rolekv_tensor k, rolekv_tensor v,
               const int32_t* keep_idx, float budget, void* k_out, void* v_out,
               int32_t* status_dev, void* stream) {
  NvtxRange nvtx("rolekv:kv_compact");
  BatchInfo bi;
  int rc = check_batch(batch, &bi);
  if (rc) return rc;
  if (!(budget > 0.f) || budget > 1.f)
    return fail(ROLEKV_ERR_INVALID_ARG, "budget %g outside (0, 1]", static_cast<double>(budget));
  if (bi.T == 0) return ROLEKV_OK;                 // no tokens: no kept rows
  if ((rc = check_compact_args(bi, k, v, keep_idx, k_out, v_out))) return rc;
  CompactArgs a;
  fill_compact(bi, batch->cu_seqlens_dev, to_fixed(budget), batch->seqlens_host, k, v, keep_idx,
               k_out, v_out, status_dev, &a);
  if (g_shrink_rows > 0) {                         // (checked-build self-test only)
    a.ext_out_rows -= g_shrink_rows;
    g_shrink_rows = 0;
  }
  if (bi.n_max == 0) return ROLEKV_OK;
  stage_begin();
  cudaError_t e = launch_compact(a, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "kv_compact");
  stage_mark(static_cast<cudaStream_t>(stream));
  return ROLEKV_OK;
}

int rolekv_compress(const rolekv_batch* batch, rolekv_tensor q_win, rolekv_tensor k,
                    rolekv_tensor v, int32_t W, int32_t pool_k, float scale,
                    const float* lse_win, const uint8_t* roles,
                    const rolekv_select_params* params, int32_t* keep_idx, void* k_out,
                    void* v_out, int32_t* kept_per_role, void* workspace,
                    size_t workspace_bytes, int32_t* status_dev, void* stream) {
  NvtxRange nvtx("rolekv:rolekv_compress");
  BatchInfo bi;
  int rc = check_batch(batch, &bi);
  if (rc) return rc;
  if (pool_k < 1 || pool_k > 15 || pool_k % 2 == 0)
    return fail(ROLEKV_ERR_UNSUPPORTED, "pool_k=%d must be odd, 1..15", pool_k);
  ScorePlan p;
  rc = plan_score(kModeSnapKV, bi, W, true, true, &p, true);
  if (rc) return rc;
  SelectArgs sa;
  if ((rc = fill_select(bi, batch, params, &sa))) return rc;
  if (bi.T == 0) {                                 // no tokens: only the zero per-role counts
    if (kept_per_role == nullptr) return ROLEKV_OK;
    sa.pool_k = pool_k;
    sa.kept_per_role = kept_per_role;
    sa.status = status_dev;
    const cudaError_t e0 = launch_select(sa, static_cast<cudaStream_t>(stream));
    return e0 == cudaSuccess ? ROLEKV_OK : cuda_fail(e0, "role_alloc_select");
  }
  if (roles == nullptr || keep_idx == nullptr) return fail(ROLEKV_ERR_INVALID_ARG, "roles and keep_idx are required");
  if ((rc = check_tensor("q_win", q_win, bi.d, bi.Hq, false, true))) return rc;
  if ((rc = check_tensor("k", k, bi.d, bi.Hkv, bi.varlen, true))) return rc;
  if ((rc = check_compact_args(bi, k, v, keep_idx, k_out, v_out))) return rc;
  if ((rc = bind_workspace(p, workspace, workspace_bytes))) return rc;
  if (bi.n_max == 0) return ROLEKV_OK;
  float* pre = reinterpret_cast<float*>(static_cast<uint8_t*>(workspace) + p.off_prepool);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  stage_begin();
  rc = run_snapkv(bi, batch->cu_seqlens_dev, q_win, k, W, scale, lse_win, pre, p, status_dev, st);
  if (rc) return rc;
  sa.scores = pre;
  sa.roles = roles;
  sa.pool_k = pool_k;
  sa.keep_idx = keep_idx;
  sa.keep_mask = nullptr;
  sa.kept_per_role = kept_per_role;
  sa.status = status_dev;
  cudaError_t e = launch_select(sa, st);
  if (e != cudaSuccess) return cuda_fail(e, "role_alloc_select");
  stage_mark(st);
  CompactArgs ca;
  fill_compact(bi, batch->cu_seqlens_dev, sa.budget_fx, batch->seqlens_host, k, v, keep_idx, k_out,
               v_out, status_dev, &ca);
  e = launch_compact(ca, st);
  if (e != cudaSuccess) return cuda_fail(e, "kv_compact");
  stage_mark(st);
  return ROLEKV_OK;
}

int snapkv_score_noalloc(const rolekv_batch* batch, rolekv_tensor q_win, rolekv_tensor k,
                         int32_t W, int32_t pool_k, float scale, const float* lse_win,
                         float* scores, float* scores_prepool, int32_t* status_dev,
                         void* stream) {
  NvtxRange nvtx("rolekv:snapkv_score_noalloc");
  BatchInfo bi;
  int rc = check_batch(batch, &bi);
  if (rc) return rc;
  if (pool_k < 1 || pool_k > 15 || pool_k % 2 == 0)
    return fail(ROLEKV_ERR_UNSUPPORTED, "pool_k=%d must be odd, 1..15", pool_k);
  ScorePlan p;
  rc = plan_score(kModeSnapKV, bi, W, lse_win == nullptr, false, &p);
  if (rc) return rc;
  if (bi.T == 0) return ROLEKV_OK;                 // no tokens: nothing to score (as snapkv_score)
  if (scores == nullptr) return fail(ROLEKV_ERR_INVALID_ARG, "scores is NULL");
  if (pool_k > 1 && scores_prepool == nullptr)
    return fail(ROLEKV_ERR_INVALID_ARG,
                "snapkv_score_noalloc with pool_k > 1 needs scores_prepool (the pre-pool output)");
  if (p.bytes > kNoAllocScratchBytes)
    return fail(ROLEKV_ERR_UNSUPPORTED,
                "batch needs %zu bytes of scratch; snapkv_score_noalloc holds at most %zu "
                "(use snapkv_score with a workspace)",
                p.bytes, kNoAllocScratchBytes);
  if ((rc = check_tensor("q_win", q_win, bi.d, bi.Hq, false, true))) return rc;
  if ((rc = check_tensor("k", k, bi.d, bi.Hkv, bi.varlen, true))) return rc;
  if (bi.n_max == 0) return ROLEKV_OK;
  void* scratch = nullptr;
  if ((rc = noalloc_scratch(&scratch))) return rc;
  // Pass 1 writes every partial slot and the normaliser kernel every row
  // before either is read, so nothing left by an earlier call is used.
  if ((rc = bind_workspace(p, scratch, kNoAllocScratchBytes))) return rc;
  float* pre = scores_prepool ? scores_prepool : scores;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  stage_begin();
  rc = run_snapkv(bi, batch->cu_seqlens_dev, q_win, k, W, scale, lse_win, pre, p, status_dev, st);
  if (rc) return rc;
  if (pool_k == 1) {
    if (pre == scores) return ROLEKV_OK;
    cudaError_t e = cudaMemcpyAsync(scores, pre, static_cast<size_t>(score_elems(bi)) * 4,
                                    cudaMemcpyDeviceToDevice, st);
    if (e != cudaSuccess) return cuda_fail(e, "copy of pre-pool scores");
    return ROLEKV_OK;
  }
  cudaError_t e = launch_maxpool(p.a, pre, scores, pool_k, st);
  if (e != cudaSuccess) return cuda_fail(e, "max-pool");
  stage_mark(st);
  return ROLEKV_OK;
}

int rolekv_checked_build(void) {
#ifdef ROLEKV_CHECKED
  return 1;
#else
  return 0;
#endif
}

int rolekv_selftest_shrink_extent(int64_t rows) {
#ifdef ROLEKV_CHECKED
  if (rows < 1 || rows > 1000000)
    return fail(ROLEKV_ERR_INVALID_ARG, "rows=%lld outside 1..1e6", static_cast<long long>(rows));
  g_shrink_rows = rows;
  return ROLEKV_OK;
#else
  (void)rows;
  return fail(ROLEKV_ERR_UNSUPPORTED, "not a checked build (librolekv_checked.so has the checks)");
#endif
}

int rolekv_selftest_score_timeout(int64_t limit_ns) {
  if (limit_ns < 1000 || limit_ns > 10000000000LL)
    return fail(ROLEKV_ERR_INVALID_ARG, "limit_ns=%lld outside 1e3..1e10", static_cast<long long>(limit_ns));
  g_timeout_test_armed = true;
  g_timeout_test_ns = static_cast<uint64_t>(limit_ns);
  return ROLEKV_OK;
}

int rolekv_set_stage_events(void* const* events, int32_t n) {
  if (n < 0 || n > kMaxStageEvents || (n > 0 && events == nullptr))
    return fail(ROLEKV_ERR_INVALID_ARG, "0..%d stage events", kMaxStageEvents);
  for (int i = 0; i < n; ++i) g_stage_events[i] = static_cast<cudaEvent_t>(events[i]);
  g_num_stage_events = n;
  return ROLEKV_OK;
}

}  // extern "C"
