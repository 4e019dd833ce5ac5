/*
 * rolekv.h -- C ABI of librolekv: the data-parallel hot path of
 * role-conditional KV-cache eviction (arXiv 2607.13205, "Adaptive Filtering of
 * the KV Cache").
 *
 * Pipeline (Algorithm 1, per layer and KV head):
 *   snapkv_score      windowed attention mass of the last W queries, GQA heads
 *                     summed, then the 1-D max-pool along the KV axis;
 *   h2o_score         the H2O accumulated mass s(t) = sum_q p_t(q) it is
 *                     compared against (Section 2);
 *   role_alloc_select per-role-bucket top-k under the budget B, split by the
 *                     role weights alpha with the single tuned knob alpha_KEY
 *                     (Section 4.1);
 *   kv_compact        gather of the kept K/V rows into a dense cache (the
 *                     compacting implementation of Section 6).
 *
 * Conventions shared by every call
 * --------------------------------
 * Units.  One unit is one (layer l, sequence s, KV head h); units are numbered
 *   u = (l * b + s) * Hkv + h.  Query head hq belongs to KV head hq / G with
 *   G = Hq / Hkv (grouped-query attention, consecutive heads share a KV head).
 * Dense and varlen batches.  With rolekv_batch.seqlens_host == NULL every
 *   sequence has n_max tokens.  Otherwise sequence s has seqlens_host[s]
 *   tokens (0 <= len <= n_max) and cu_seqlens_dev must hold, on the device, the
 *   b+1 prefix sums 0, len0, len0+len1, ... (int32).
 * Tensors.  A rolekv_tensor is a device pointer to bf16 elements plus element
 *   strides for (layer, sequence, head, token); the last (head-dim) axis is
 *   contiguous.  Element (l, s, h, t, :) lives at
 *     ptr + l*s_layer + s*s_seq + h*s_head + t*s_tok            (dense)
 *     ptr + l*s_layer + (cu[s] + t)*s_tok + h*s_head            (varlen)
 *   The pointer must be 16-byte aligned and every stride a multiple of 8
 *   elements; s_layer and s_seq must be multiples of s_tok, and s_head either
 *   a multiple of s_tok or small enough that all heads fit in one token row
 *   ((H-1)*s_head + d <= s_tok).  [L][b][H][n][d] and varlen [L][T][H][d]
 *   contiguous tensors both qualify.
 * Score arrays (fp32).  Dense: [L][b][Hkv][n_max].  Varlen: [L][Hkv][T],
 *   sequence s at columns cu[s] .. cu[s+1]-1.
 * Role arrays (uint8, one label per token, shared by all layers and heads).
 *   Dense: [b][n_max].  Varlen: [T].
 * Kept-index arrays (int32).  Sequence s has a row of K_s =
 *   rolekv_kept_rows(len_s, B, kept_extra) slots: its ceil(B*len_s) budget
 *   plus the batch's kept_extra, at most len_s (kept_extra is 0 except for the
 *   ceiling policy, whose total may exceed the budget).  Dense: [L][b][Hkv][K],
 *   K = rolekv_kept_rows(n_max, B, kept_extra).  Varlen: [L][Hkv][Ktot],
 *   sequence s at offset cu_kept[s] = sum of K_s' for s' < s.  Kept positions
 *   are written in ascending order; the slots after the last kept position
 *   (fewer eligible tokens than the budget, or the unused part of kept_extra)
 *   hold -1.  kv_compact, decode_attention and rolekv_compress use the same
 *   rows for the same batch and budget.
 * Batches without tokens.  When n_max is 0 or every sequence is empty, the
 *   buffers sized by tokens or kept slots are empty and may be NULL; the
 *   calls still write what is not empty: zero per-role kept counts and zero
 *   decode outputs.
 * Ownership.  The caller owns every buffer; the library allocates, frees and
 *   synchronises nothing.  Every call enqueues work on `stream` (a
 *   cudaStream_t; NULL means the legacy default stream) and returns at once.
 * Errors.  Argument problems are detected on the host before anything is
 *   enqueued and return a ROLEKV_ERR_* code; rolekv_last_error() then gives a
 *   one-line description.  Conditions seen on the device (non-finite scores,
 *   an out-of-range kept index, a wait that ran out) never trap: they are
 *   OR-ed into the optional int32 *status_dev word (ROLEKV_STATUS_* bits),
 *   which the caller clears and reads.
 */
#ifndef ROLEKV_H
#define ROLEKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ROLEKV_OK 0
#define ROLEKV_ERR_INVALID_ARG 1
#define ROLEKV_ERR_UNSUPPORTED 2
#define ROLEKV_ERR_WORKSPACE 3
#define ROLEKV_ERR_CUDA 4

#define ROLEKV_STATUS_NONFINITE 1   /* a NaN score was seen by the selector    */
#define ROLEKV_STATUS_BAD_INDEX 2   /* kv_compact met an index >= the length  */
#define ROLEKV_STATUS_TIMEOUT 4     /* a bounded device wait gave up          */
#define ROLEKV_STATUS_BOUNDS 8      /* checked build: an access fell outside the
                                       extent the call's shapes give its buffer
                                       and was skipped                         */

#define ROLEKV_POLICY_ROLE_QUOTA 0  /* the combined method (Section 4.1)       */
#define ROLEKV_POLICY_GLOBAL 1      /* plain top-k, optional role ban (Sec. 4) */
#define ROLEKV_POLICY_FAIR 2        /* equal retention rate per role (Sec. 5)  */
#define ROLEKV_POLICY_SLACK 3       /* slack of saturated buckets by score     */
#define ROLEKV_POLICY_CEIL 4        /* Algorithm 1's ceilings taken literally  */

#define ROLEKV_MAX_ROLES 8
#define ROLEKV_SELECT_MAX_N 262144  /* largest sequence role_alloc_select takes */

typedef struct rolekv_tensor {
  const void* ptr;
  int64_t s_layer, s_seq, s_head, s_tok;
} rolekv_tensor;

typedef struct rolekv_batch {
  int32_t L, b, Hq, Hkv, d;
  int32_t n_max;
  const int32_t* seqlens_host;   /* [b] on the host, or NULL (dense)          */
  const int32_t* cu_seqlens_dev; /* [b+1] on the device, varlen only          */
  int32_t kept_extra;            /* kept-row slots beyond ceil(B*n), >= 0;
                                    ROLEKV_POLICY_CEIL needs at least the
                                    number of weighted roles - 1; 0 otherwise */
} rolekv_batch;

/* Role-conditional allocation parameters (Section 4.1, Algorithm 1).
 *   alpha[r]   weight of role r (>= 0); alpha[key_role] is replaced by
 *              alpha_key, the method's one tuned knob (0 bans KEY, 0.02 is the
 *              paper's safe default).
 *   budget     B in (0, 1]; a sequence of n tokens keeps ceil(B*n) tokens
 *              (B is taken to 1e-6 fixed point so the ceiling is exact).
 *   policy     ROLEKV_POLICY_ROLE_QUOTA: bucket r keeps its share
 *              alpha_r / sum(alpha of eligible buckets) of the budget, a bucket
 *              being eligible when alpha_r > 0, it holds tokens and is not
 *              banned; a bucket whose share reaches its size keeps everything
 *              and its slack goes to the others in proportion to alpha
 *              (repeated water-filling), and the integer quotas are floors plus
 *              largest remainders (ties to the lower role id), so they sum to
 *              exactly min(ceil(B*n), eligible tokens).
 *              ROLEKV_POLICY_GLOBAL: one bucket of all non-banned tokens, top
 *              min(ceil(B*n), eligible) by score (plain H2O / SnapKV top-k;
 *              with ban_mask it is the counterfactual 'No-X' ban of Section 4).
 *              ROLEKV_POLICY_FAIR: the fair-eviction baseline of Section 5
 *              (equal retention rate per role): as ROLE_QUOTA with every
 *              non-banned role weighted by its token count; alpha is unused.
 *              ROLEKV_POLICY_SLACK: the other reading of Algorithm 1's
 *              "redistribute unused budget from saturated buckets": one
 *              round of the ROLE_QUOTA split (no water-filling), each quota
 *              capped at its bucket's size, then the slots that saturated
 *              buckets leave go to the highest-scoring tokens of the
 *              eligible buckets not kept yet (ties to the lower index); the
 *              total is the same min(ceil(B*n), eligible tokens).
 *              ROLEKV_POLICY_CEIL: Algorithm 1's "top ceil(alpha_r B n_kv)
 *              per bucket" taken literally: the ROLE_QUOTA water-filling of
 *              saturated buckets, then each unsaturated bucket keeps the
 *              ceiling of its share instead of floor plus largest remainder.
 *              The total lies between min(ceil(B*n), eligible) and that plus
 *              (unsaturated buckets - 1), so the batch's kept_extra must be at
 *              least (roles with a positive weight, not banned) - 1, else the
 *              call returns ROLEKV_ERR_INVALID_ARG.
 *   ban_mask   bit r set: role r keeps nothing.
 *   keep_last  recency floor (SnapKV's observation window, Section 7): the
 *              last R = min(keep_last, n, ceil(B*n)) tokens of each sequence
 *              are kept whatever their score and role; the other
 *              ceil(B*n) - R slots are split as above over the earlier tokens,
 *              whose roles alone are counted.  0: no floor.
 * Within a bucket the highest scores win and equal scores go to the lower
 * token index. */
typedef struct rolekv_select_params {
  int32_t n_roles;               /* 1 .. ROLEKV_MAX_ROLES                     */
  float alpha[ROLEKV_MAX_ROLES];
  int32_t key_role;              /* -1: no override                           */
  float alpha_key;
  float budget;
  int32_t policy;
  uint32_t ban_mask;
  int32_t keep_last;             /* >= 0                                      */
} rolekv_select_params;

/* Number of kept slots of an n-token sequence at budget B: ceil(B*n) with B in
 * 1e-6 fixed point; -1 if B is outside (0, 1] or n < 0. */
int64_t rolekv_kept_count(int64_t n, float budget);

/* Width of an n-token sequence's kept-index row: min(n, rolekv_kept_count(n,
 * budget) + kept_extra); -1 for a budget outside (0, 1], n < 0 or
 * kept_extra < 0. */
int64_t rolekv_kept_rows(int64_t n, float budget, int32_t kept_extra);

/* Bytes of device workspace snapkv_score / h2o_score / rolekv_compress need for
 * this batch (op: 0 snapkv_score, 1 h2o_score, 2 rolekv_compress; W the SnapKV
 * window).  The workspace is caller-owned scratch, 256-byte aligned, reusable
 * across calls on the same stream; its contents need no initialisation. */
int rolekv_workspace_size(int op, const rolekv_batch* batch, int32_t W, size_t* bytes);

/* SnapKV windowed score (Section 2; Section 4 'SnapKV mechanism'; Algorithm 1,
 * windowed mass and pooling steps).  With pool_k == 1 and no scores_prepool
 * the pre-pool score is written straight to `scores` (no pool kernel).
 *   q_win   bf16 window queries, [L][b][Hq][W][d] addressed by its strides
 *           (dense in the sequence axis even for varlen batches); row i of a
 *           sequence of n tokens is the query at position n - W_eff + i,
 *           W_eff = min(W, n); rows i >= W_eff are ignored.
 *   k       bf16 keys of the batch.
 *   W       window length, a multiple of 8 with W*G <= 256.
 *   pool_k  odd max-pool width, 1 .. 15 (1 = no pooling).
 *   scale   softmax scale; <= 0 selects 1/sqrt(d).
 *   lse_win optional fp32 [L][b][Hq][W]: the natural-log softmax normaliser of
 *           each window row over its causal keys (the prefill attention's own
 *           LSE).  NULL: computed here (two passes over K).
 *   scores  fp32 score array, receives the pooled score s~(t).
 *   scores_prepool  optional fp32 score array for s(t) before pooling.
 * s(t) = sum over the G query heads of the KV head and the W_eff window rows of
 * softmax(scale * q K^T) at key t, causal inside the window; the pool is stride
 * 1, same length, truncated at the sequence ends.  d must be 64 or 128. */
int snapkv_score(const rolekv_batch* batch, rolekv_tensor q_win, rolekv_tensor k, int32_t W,
                 int32_t pool_k, float scale, const float* lse_win, float* scores,
                 float* scores_prepool, void* workspace, size_t workspace_bytes,
                 int32_t* status_dev, void* stream);

/* snapkv_score without a workspace (the paper has no counterpart; this is a
 * deployment convenience of this library).  Some callers cannot allocate
 * device memory at the point where they score: an inference server whose
 * memory manager has already handed all of HBM to the KV cache and forbids
 * further allocations, a plugin that is given only its input and output
 * buffers, or a latency-critical path where cudaMalloc's device-wide
 * synchronisation is not acceptable.  This call takes the same inputs and
 * outputs as snapkv_score and keeps its scratch (the pass-1 partial row
 * statistics and the per-row normalisers) in a static device array of
 * 64 MiB that every GPU loading this library reserves until the process
 * exits; it calls no cudaMalloc, cudaFree or other allocating routine.
 *   Limits: batches whose scratch would exceed 64 MiB are rejected with
 *   ROLEKV_ERR_UNSUPPORTED (about 9 MiB for 32 layers x 4 x 8 KV heads at
 *   32768 tokens); with pool_k > 1, scores_prepool is required, because the
 *   pre-pool scores are an output here, not scratch.
 *   Set-up: every call looks up the array's device address in the current
 *   context (cudaGetSymbolAddress, a cheap runtime query), so a context that
 *   was reset and made again gets its own array; the first call on a device
 *   also loads the library's device code there, so make it before any
 *   stream capture.
 *   Empty batches (no tokens) return ROLEKV_OK without touching any buffer,
 *   as snapkv_score does.
 *   Sharing: every call on a device uses the same array and leaves its
 *   contents behind; each call overwrites all it reads, so nothing needs
 *   clearing, but calls that overlap on the GPU (other streams, other host
 *   threads) race on the array -- order them on one stream. */
int snapkv_score_noalloc(const rolekv_batch* batch, rolekv_tensor q_win, rolekv_tensor k,
                         int32_t W, int32_t pool_k, float scale, const float* lse_win,
                         float* scores, float* scores_prepool, int32_t* status_dev,
                         void* stream);

/* Quest one-shot analogue (Section 5, "Query-aware baseline"): the mean query
 * qbar of the window rows (the last W_eff = min(W, n) positions of the G query
 * heads of each KV head; q_win as for snapkv_score) scores every page of `page`
 * consecutive tokens of a sequence by the key bound
 *   sum_i max(qbar_i * min_t k_ti, qbar_i * max_t k_ti)   (t over the page),
 * an upper bound on qbar . k_t for every token of the page; the last page of a
 * sequence may be short.  Every token's entry of `scores` (the layout of
 * snapkv_score's output) is its page's bound, so role_alloc_select (pool_k 1,
 * GLOBAL for Quest's plain page top-k, ties to the lower index keep whole pages
 * in bound order) runs on it as on any score.
 * d must be 64 or 128; 1 <= page <= 4096; W >= 1.  No workspace. */
int quest_score(const rolekv_batch* batch, rolekv_tensor q_win, rolekv_tensor k, int32_t W,
                int32_t page, float* scores, void* stream);

/* One decode step of attention through a cache of kept rows (Section 6: the
 * compacted cache realises the 1-B memory and decode-time reduction).  For
 * every (layer, sequence, KV head) and each of its G query heads,
 *   out_g = sum_j softmax_j(scale * q_g . k_j) v_j
 * over the unit's rows j < rolekv_kept_rows(n, budget, kept_extra) of k_cache /
 * v_cache, skipping the rows whose keep_idx entry is -1 (padding).
 *   q        bf16 decode queries, one token per sequence: [L][b][Hq][d]
 *            (s_tok is ignored).
 *   k_cache, v_cache  bf16 cache rows: kv_compact's output (dense
 *            [L][b][Hkv][K][d], varlen [L][Hkv][Ktot][d]: token index =
 *            kept rows of the earlier sequences + j), or, with budget 1 and
 *            keep_idx NULL, the full cache in its own layout (varlen
 *            [L][T][Hkv][d]).
 *   keep_idx the kept index rows role_alloc_select wrote, or NULL (all valid).
 *   scale    <= 0: 1/sqrt(d).
 *   out      fp32 [L][b][Hq][d], contiguous.
 *   workspace  rolekv_decode_workspace_size() bytes (partials of the split
 *            rows), caller-owned, no initialisation needed.
 *   status_dev optional int32 status word (ROLEKV_STATUS_TIMEOUT).
 * d must be 64 or 128 and G <= 8; a unit with no valid row gives zeros. */
int rolekv_decode_workspace_size(const rolekv_batch* batch, float budget, size_t* bytes);
int decode_attention(const rolekv_batch* batch, rolekv_tensor q, rolekv_tensor k_cache,
                     rolekv_tensor v_cache, const int32_t* keep_idx, float budget, float scale,
                     float* out, void* workspace, size_t workspace_bytes, int32_t* status_dev,
                     void* stream);

/* H2O accumulated attention mass (Section 2): s(t) = sum over the G query heads
 * of the KV head and every causal query position q >= t of p_t(q).
 *   q       bf16 prefill queries of every position: dense [L][b][Hq][n][d] or
 *           varlen [L][T][Hq][d], addressed by its strides.
 *   scale   softmax scale; <= 0 selects 1/sqrt(d).
 *   lse     optional fp32 natural-log softmax normaliser of every query row
 *           over its causal keys (the softmax_lse a prefill attention already
 *           produces): dense [L][b][Hq][n_max], varlen [L][Hq][T] (sequence s
 *           at columns cu[s] .. cu[s+1]-1), 4-byte aligned.  Given, the keys
 *           are read and multiplied once (pass 2 only); NULL: the normalisers
 *           are computed here, in a first pass over the same key tiles.
 *   scores  fp32 score array.  No pooling (the H2O score has none).  Each
 *           score is a sum of per-query-block parts added atomically, in an
 *           order that varies between runs (about 1e-7 relative).
 * d must be 64 or 128 and G <= 8. */
int h2o_score(const rolekv_batch* batch, rolekv_tensor q, rolekv_tensor k, float scale,
              const float* lse, float* scores, void* workspace, size_t workspace_bytes,
              int32_t* status_dev, void* stream);

/* Role-conditional allocation and per-bucket top-k (Section 4.1, Algorithm 1).
 *   scores        fp32 score array (pooled SnapKV, H2O, or any score).
 *   roles         uint8 role array; labels >= n_roles belong to no bucket.
 *   pool_k        odd width of a max-pool applied to `scores` first (1 = none);
 *                 lets a caller pass pre-pool SnapKV scores.
 *   keep_idx      int32 kept-index array (ascending positions, -1 padded).
 *   keep_mask     optional uint8 array in the score layout: 1 kept, 0 evicted.
 *   kept_per_role optional int32 [units][n_roles]: kept tokens per role.
 * Sequences longer than ROLEKV_SELECT_MAX_N are rejected (ERR_UNSUPPORTED).
 * Rows of up to 40960 tokens keep their pooled keys in shared memory; longer
 * rows recompute them from the score row on each pass (the same kept set,
 * more reads of the scores from L2). */
int role_alloc_select(const rolekv_batch* batch, const float* scores, const uint8_t* roles,
                      const rolekv_select_params* params, int32_t pool_k, int32_t* keep_idx,
                      uint8_t* keep_mask, int32_t* kept_per_role, int32_t* status_dev,
                      void* stream);

/* Gather-compaction of the retained rows (Section 6, compacting
 * implementation): k_out[u][j] = K[u][keep_idx[u][j]] and the same for V, for
 * every kept slot j; slots holding -1 become zero rows.  k_out / v_out are
 * dense bf16 [L][b][Hkv][K][d] (varlen: [L][Hkv][Ktot][d]) with the kept-index
 * layout of `budget` and the batch's kept_extra.  d must be a multiple of 8,
 * at most 256.  k and v may also point into pinned (page-locked, device-
 * mapped) host memory: the kernel then reads only the kept rows across the
 * host link, which moves B of the cache instead of all of it. */
int kv_compact(const rolekv_batch* batch, rolekv_tensor k, rolekv_tensor v,
               const int32_t* keep_idx, float budget, void* k_out, void* v_out,
               int32_t* status_dev, void* stream);

/* The whole path in one call: snapkv_score (pre-pool scores kept in the
 * workspace), role_alloc_select with the pool fused into its load, and
 * kv_compact.  Arguments as in the calls above; the pooled scores are not
 * written out. */
int rolekv_compress(const rolekv_batch* batch, rolekv_tensor q_win, rolekv_tensor k,
                    rolekv_tensor v, int32_t W, int32_t pool_k, float scale,
                    const float* lse_win, const uint8_t* roles,
                    const rolekv_select_params* params, int32_t* keep_idx, void* k_out,
                    void* v_out, int32_t* kept_per_role, void* workspace,
                    size_t workspace_bytes, int32_t* status_dev, void* stream);

/* Optional per-kernel timing for callers that profile the path.  After this
 * call every later call made on the same thread records events[i]
 * (cudaEvent_t, created by the caller) on its stream right after its i-th
 * kernel launch, for i < n (n <= 8; n = 0 switches it off).  Kernel order:
 * snapkv_score / rolekv_compress: pass 1 (absent when lse_win is given), the
 * window normalisers, pass 2, then the pool (snapkv_score with pool_k > 1) or
 * the selector and the compaction (rolekv_compress); h2o_score: pass 1,
 * pass 2; role_alloc_select and kv_compact: their one kernel.  The setting
 * is per thread and holds no device memory. */
int rolekv_set_stage_events(void* const* events, int32_t n);

/* One-line description of the last error returned on this thread. */
const char* rolekv_last_error(void);

/* Library version string. */
const char* rolekv_version(void);

/* Diagnostic (no counterpart in the paper): runs the bounded device wait the
 * kernels use on a barrier phase that nothing completes, so that it gives up
 * after limit_ns nanoseconds (0 .. 1e10) and ORs ROLEKV_STATUS_TIMEOUT into
 * *status_dev (device int32, required); the kernel then returns normally.
 * It lets a caller check, without a fault, that a stuck wait is reported and
 * the context stays usable. */
int rolekv_selftest_wait(int64_t limit_ns, int32_t* status_dev, void* stream);

/* Diagnostic (no counterpart in the paper): arms the next two-pass SnapKV
 * score (snapkv_score or rolekv_compress without lse_win) made on the calling
 * thread so that the persistent score kernel's per-unit meeting point, where
 * a unit's key chunks wait for each other between the two passes, waits for
 * one arrival more than there are chunks -- one that never comes -- with a
 * limit of limit_ns nanoseconds (1e3 .. 1e10) instead of the usual 2 s.  That
 * call then gives up at the meeting point, ORs ROLEKV_STATUS_TIMEOUT into its
 * status word, drains its copies and tensor-core work, frees its tensor
 * memory and returns; its scores are not valid.  The arming is used up by
 * that one call.  It lets a caller check, without a fault, that the real
 * kernel's abort path reports the stuck wait and leaves the device usable. */
int rolekv_selftest_score_timeout(int64_t limit_ns);

/* Checked build (no counterpart in the paper).  The library can be built a
 * second time with -DROLEKV_CHECKED (librolekv_checked.so beside
 * librolekv.so, same entry points).  Every kernel there checks each global
 * load or store whose address it computes from run-time data (kept indices,
 * sequence offsets, unit and chunk offsets, strides) against the extent the
 * call's shapes and strides give that buffer.  An access outside it is
 * skipped and ROLEKV_STATUS_BOUNDS is OR-ed into the status word: a kernel
 * bug then shows up as a status bit and a wrong output, not as a memory
 * fault.  Loads and stores through TMA tensor maps are bounded by the maps
 * themselves and are not checked again.  The checks cost time; the plain
 * build has none.
 *
 * rolekv_checked_build() returns 1 in the checked build and 0 in the plain
 * one. */
int rolekv_checked_build(void);

/* Diagnostic for the checked build (no counterpart in the paper): the next
 * kv_compact call made on the calling thread takes its output extent as
 * `rows` kept rows smaller than its shapes give (1 .. 1e6), so that the
 * checks on the last rows fire although every access is inside the real
 * buffer.  That call skips those rows' stores (their output is left as it
 * was) and ORs ROLEKV_STATUS_BOUNDS into its status word.  The arming is used
 * up by that one call.  It lets a caller see that the checks report and skip
 * without provoking a single out-of-range access.  Returns
 * ROLEKV_ERR_UNSUPPORTED in the plain build. */
int rolekv_selftest_shrink_extent(int64_t rows);

#ifdef __cplusplus
}
#endif
#endif /* ROLEKV_H */
