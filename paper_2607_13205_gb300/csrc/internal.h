// Internal interfaces between the C-ABI layer and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "rolekv.h"

namespace rolekv {

enum { kModeSnapKV = 0, kModeH2O = 1 };

// Every device-side wait is bounded by this much wall time (globaltimer, ns);
// when it runs out the kernel records ROLEKV_STATUS_TIMEOUT and unwinds.
constexpr uint64_t kWaitLimitNs = 2000000000ull;

// Everything the two attention passes need, passed by value to the kernels.
struct ScoreArgs {
  int32_t L, b, G, Hkv, d, n_max;
  int32_t varlen;
  int64_t T;                        // packed tokens (varlen score layout)
  const int32_t* cu_seqlens;        // device, varlen only
  int32_t mode;                     // kModeSnapKV / kModeH2O
  int32_t W;                        // SnapKV window
  int32_t P;                        // positions per query block (SnapKV: W)
  int32_t nrows;                    // G * P rows in a query block
  int32_t nrows_pad;                // 128 or 256
  int32_t n_units;
  int64_t k_layer, k_seq, k_head, k_tok;
  int64_t q_layer, q_seq, q_head, q_tok;
  float c1;                         // softmax scale * log2(e)
  int32_t chunk_tiles;              // SnapKV: 128-key tiles per CTA
  int32_t n_chunks;                 // SnapKV: CTAs per unit
  int32_t nrb_max;                  // H2O: query blocks per unit (largest sequence)
  float2* partials;                 // SnapKV pass 1: [unit][chunk][256] (max2, sum)
  float* lse2;                      // [unit][query block][256] log2-domain normalisers
  float* prepool;                   // score output before pooling
  int32_t* status;
  // element extents the call's shapes give these buffers (checked build)
  int64_t ext_scores;               // prepool and the pooled scores
  int64_t ext_partials;
  int64_t ext_lse2;
  int64_t ext_lse_win;              // a caller-supplied window LSE
};

cudaError_t launch_attn_pass(int pass, int d, const CUtensorMap& kmap, const CUtensorMap& qmap,
                             const ScoreArgs& a, int grid, cudaStream_t stream);

// The SnapKV score in one persistent, cooperative launch: (unit, chunk of
// key tiles) items are dealt round-robin to the CTAs; each runs pass 1 on its
// chunk, meets the unit's other chunks at a bounded arrival counter, forms
// the exact normalisers from their partials and runs pass 2 on the same (now
// L2-resident) tiles.
struct FusedArgs {
  ScoreArgs s;                      // s.n_chunks = chunks per unit, s.chunk_tiles = tiles per chunk
  int32_t* work;                    // [1 + u]: chunks of unit u done with pass 1 ([0] unused)
  int32_t n_items;
  int32_t single;                   // 1: pass 2 only; SnapKV normalisers given in s.lse2,
                                    // H2O ones in h2o_lse
  const float* h2o_lse;             // H2O, single: natural-log LSE of every query row
                                    // (dense [L][b][Hq][n_max], varlen [L][Hq][T])
  uint64_t wait_ns;                 // limit of the per-unit meeting point's wait
  int32_t hold;                     // arrivals the meeting point waits for beyond the
                                    // unit's chunks (0; 1 only in the timeout self-test)
  int64_t ext_h2o_lse;              // elements of h2o_lse (checked build)
};

cudaError_t launch_snapkv_fused(int d, const CUtensorMap& kmap, const CUtensorMap& qmap,
                                const FusedArgs& a, cudaStream_t stream);
cudaError_t launch_snapkv_lse(const ScoreArgs& a, const float* lse_win, cudaStream_t stream);
cudaError_t launch_maxpool(const ScoreArgs& a, const float* in, float* out, int pool_k,
                           cudaStream_t stream);

// Selection ------------------------------------------------------------------

struct SelectArgs {
  int32_t L, b, Hkv, n_max;
  int32_t varlen;
  int64_t T;                        // packed tokens
  int64_t Ktot;                     // packed kept slots (varlen)
  int32_t K_dense;                  // kept slots per unit (dense)
  const int32_t* cu_seqlens;
  int32_t n_units;
  const float* scores;
  const uint8_t* roles;
  int32_t pool_k;
  int32_t n_roles;
  int64_t alpha_fx[ROLEKV_MAX_ROLES];   // fixed-point weights, 0 for banned roles
  int64_t budget_fx;
  int32_t kept_extra;                   // kept-row width beyond ceil(B n)
  int32_t policy;
  uint32_t ban_mask;
  int32_t keep_last;                    // recency floor (tokens), 0 = none
  int32_t* keep_idx;
  uint8_t* keep_mask;
  int32_t* kept_per_role;
  int32_t* status;
  // element extents (checked build): scores and keep_mask, roles, keep_idx
  int64_t ext_scores, ext_roles, ext_keep;
};

cudaError_t launch_select(const SelectArgs& a, cudaStream_t stream);

// Quest one-shot analogue ----------------------------------------------------

struct QuestArgs {
  int32_t L, b, G, Hkv, d, n_max;
  int32_t varlen;
  int64_t T;
  const int32_t* cu_seqlens;
  int32_t n_units;
  int32_t W;                        // window rows per head averaged into the query
  int32_t page;                     // tokens per page
  const uint16_t* q;                // window queries (bf16 bits), SnapKV layout
  int64_t q_layer, q_seq, q_head, q_tok;
  const uint16_t* k;
  int64_t k_layer, k_seq, k_head, k_tok;
  float* scores;
  // element extents (checked build); quest_score has no status word, so an
  // access outside them is skipped without a report
  int64_t ext_scores, ext_q, ext_k;
};

cudaError_t launch_quest(const QuestArgs& a, cudaStream_t stream);

// Decode attention through the (compacted) cache -----------------------------

struct DecodeArgs {
  int32_t L, b, G, Hkv, d, n_max;
  int32_t varlen;
  const int32_t* cu_seqlens;
  int32_t n_units;
  int64_t budget_fx;                // rows of a sequence: kept_rows(n, budget_fx, kept_extra)
  int32_t kept_extra;
  int64_t Ktot;                     // packed rows per (layer, head), varlen
  int32_t K_dense;                  // rows per unit, dense
  const uint16_t* q;                // decode queries [L][b][Hq][d] (strides below)
  int64_t q_layer, q_seq, q_head;
  const uint16_t* k;
  int64_t k_layer, k_seq, k_head, k_tok;
  const uint16_t* v;
  int64_t v_layer, v_seq, v_head, v_tok;
  const int32_t* keep_idx;          // -1 marks an empty slot; NULL: every row valid
  float c1;                         // scale * log2(e)
  int32_t rows_per_split;
  int32_t n_splits;
  float* part;                      // [unit][split][G][d + 2]: o (unnormalised), max2, sum
  float* out;                       // fp32 outputs
  int64_t o_layer, o_seq, o_head;
  int32_t* status;
  // element extents (checked build)
  int64_t ext_q, ext_k, ext_v, ext_keep, ext_part, ext_out;
  int32_t k_tma;                    // K stages through the tensor map (swizzled halves)
  int32_t v_tma;                    // V stages through the tensor map (strided rows)
};

// kmap: a tensor map over K's token rows (box: 64 rows x 64 columns, 128-byte
// swizzle), used when a.k_tma is set; vmap: one over V's token rows (box: 64
// rows x d, no swizzle), used when a.v_tma is set (V rows strided, as in a
// packed varlen cache).
cudaError_t launch_decode(const DecodeArgs& a, const CUtensorMap& kmap, const CUtensorMap& vmap,
                          cudaStream_t stream);
cudaError_t launch_selftest_wait(uint64_t limit_ns, int32_t* status, cudaStream_t stream);

// Compaction -----------------------------------------------------------------

struct CompactArgs {
  int32_t L, b, Hkv, d, n_max;
  int32_t varlen;
  int64_t Ktot;
  int32_t K_dense;
  int32_t K_max;                    // widest kept row (grid sizing)
  int64_t budget_fx;
  int32_t kept_extra;
  const int32_t* cu_seqlens;
  int32_t n_units;
  const uint16_t* k;
  const uint16_t* v;
  int64_t k_layer, k_seq, k_head, k_tok;
  int64_t v_layer, v_seq, v_head, v_tok;
  const int32_t* keep_idx;
  uint16_t* k_out;
  uint16_t* v_out;
  int32_t* status;
  // element extents (checked build): K, V, kept slots, output rows
  int64_t ext_k, ext_v, ext_keep, ext_out_rows;
};

cudaError_t launch_compact(const CompactArgs& a, cudaStream_t stream);

// Shared helpers (host and device) ------------------------------------------

constexpr int64_t kFixedOne = 1000000;

__host__ __device__ inline int64_t kept_slots(int64_t n, int64_t budget_fx) {
  return (budget_fx * n + kFixedOne - 1) / kFixedOne;
}

// Width of an n-token sequence's kept row: ceil(B n) slots plus `extra` (room
// for the ceiling split's overshoot), at most n.
__host__ __device__ inline int64_t kept_rows(int64_t n, int64_t budget_fx, int32_t extra) {
  const int64_t k = kept_slots(n, budget_fx) + extra;
  return k < n ? k : n;
}

}  // namespace rolekv
