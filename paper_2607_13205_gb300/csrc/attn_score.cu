// Attention-mass scores on the tensor cores (sm_103a): the SnapKV windowed
// mass (Section 2; Section 4 'SnapKV mechanism'; Algorithm 1, windowed-mass
// step) and the H2O accumulated mass s(t) = sum_q p_t(q) (Section 2).
//
// Both are column sums of a causal softmax, s(t) = sum_j exp(S_jt - lse_j),
// over a set of query rows j (the G heads of a KV head times the last W
// positions, or times every position).  The exact normaliser lse_j is needed
// before any column can be summed, so the keys are visited twice:
//
//   pass 1 (rowstats): S = Q K^T with query rows on the TMEM lanes; each
//     epilogue thread owns a row and keeps its running max and sum of exp2.
//   pass 2 (colsum):   S^T = K Q^T with keys on the TMEM lanes; each epilogue
//     thread owns a key and sums exp2(S c - lse2_j) over the rows
//     thread-locally, so no cross-thread reduction is needed.  In the
//     persistent kernel the normalisers enter the accumulator through a ninth
//     MMA k-step (keys x ones against rows x -lse2_j / c1), so the epilogue
//     loads no per-row value from shared memory.
//
// In both passes one producer warp streams 128-key K tiles and 256-row query
// blocks into 128-byte-swizzled shared memory with TMA, one warp issues
// tcgen05.mma (bf16 operands, fp32 accumulators in tensor memory, two
// accumulator buffers) and sixteen epilogue warps drain the accumulators with
// tcgen05.ld.  Every wait is an mbarrier wait bounded in time.
//
// snapkv_fused_kernel runs both passes in one persistent launch, for SnapKV
// (items = chunks of a unit's keys; the chunks of a unit exchange their row
// statistics through global memory between the passes) and for H2O (items =
// query blocks; a block's normalisers are its own, so they stay on chip).
// attn_pass_kernel runs one pass per launch (the no-workspace SnapKV call).
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <type_traits>

#include "device_common.cuh"
#include "internal.h"

namespace rolekv {
namespace {

constexpr int kTileKeys = 128;
constexpr int kEpiWarps = 16;                 // four per SM sub-partition
constexpr int kParts = kEpiWarps / 4;         // epilogue warps sharing a TMEM lane quadrant
constexpr int kProducerWarp = kEpiWarps;
constexpr int kMmaWarp = kEpiWarps + 1;
constexpr int kThreads = (kEpiWarps + 2) * 32;
constexpr int kRowsMax = 256;
constexpr uint32_t kTmemCols = 512;
constexpr float kLog2e = 1.4426950408889634f;

enum { kPassRowstats = 0, kPassColsum = 1 };

template <int D, int PASS>
struct Cfg {
  static constexpr int kHalves = D / 64;                 // 128-byte swizzle atoms along d
  static constexpr int kKSteps = D / 16;                 // MMA K steps of 16
  static constexpr int kKTileBytes = kTileKeys * D * 2;  // one 128-key tile
  static constexpr int kQSlotBytes = kRowsMax * D * 2;   // one 256-row query block
  static constexpr int kKHalfBytes = kTileKeys * 128;
  static constexpr int kQHalfBytes = kRowsMax * 128;
  // every CTA keeps one query block and streams key tiles
  static constexpr int SQ = 1;
  static constexpr int SK = 4;
  static constexpr int kQOff = 0;
  static constexpr int kKOff = kQOff + SQ * kQSlotBytes;
  static constexpr int kLseOff = kKOff + SK * kKTileBytes;
  static constexpr int kPosOff = kLseOff + SQ * kRowsMax * 4;
  static constexpr int kRedOff = kPosOff + SQ * kRowsMax * 4;
  static constexpr int kMergeOff = kRedOff + (kParts - 1) * kTileKeys * 4;
  static constexpr int kBarOff = kMergeOff + kParts * kRowsMax * 8;
  static constexpr int kNumBars = 2 * SK + 2 * SQ + 4 + 3;
  static constexpr int kMiscOff = kBarOff + kNumBars * 8;
  static constexpr int kBytes = kMiscOff + 16;
  static constexpr int kSmemAlloc = kBytes + 1024;       // room to align the base to 1 KB
};

struct Shared {
  uint8_t* q;
  uint8_t* k;
  float* lse;
  int32_t* pos;
  float* red;
  float2* merge;
  uint64_t* k_full;
  uint64_t* k_empty;
  uint64_t* q_full;
  uint64_t* q_empty;
  uint64_t* acc_full;
  uint64_t* acc_empty;
  uint64_t* red_full;
  uint64_t* red_empty;
  uint64_t* drain;
  uint32_t* tmem_base;
  volatile int* abort_flag;
};

template <int D, int PASS>
__device__ __forceinline__ Shared carve(uint8_t* raw) {
  using C = Cfg<D, PASS>;
  const uint32_t a = smem_u32(raw);
  uint8_t* base = raw + ((1024u - (a & 1023u)) & 1023u);
  Shared s;
  s.q = base + C::kQOff;
  s.k = base + C::kKOff;
  s.lse = reinterpret_cast<float*>(base + C::kLseOff);
  s.pos = reinterpret_cast<int32_t*>(base + C::kPosOff);
  s.red = reinterpret_cast<float*>(base + C::kRedOff);
  s.merge = reinterpret_cast<float2*>(base + C::kMergeOff);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + C::kBarOff);
  s.k_full = bars;
  s.k_empty = bars + C::SK;
  s.q_full = bars + 2 * C::SK;
  s.q_empty = bars + 2 * C::SK + C::SQ;
  s.acc_full = bars + 2 * C::SK + 2 * C::SQ;
  s.acc_empty = s.acc_full + 2;
  s.red_full = s.acc_full + 4;
  s.red_empty = s.acc_full + 5;
  s.drain = s.acc_full + 6;
  s.tmem_base = reinterpret_cast<uint32_t*>(base + C::kMiscOff);
  s.abort_flag = reinterpret_cast<volatile int*>(base + C::kMiscOff + 4);
  return s;
}

// ---------------------------------------------------------------- geometry --

struct Unit {
  int l, s, h;
  int n;            // keys (= tokens) of the sequence
  int64_t tok0;     // first token of the sequence in the packed token axis
};

__device__ __forceinline__ Unit decode_unit(const ScoreArgs& a, int u) {
  Unit r;
  r.h = u % a.Hkv;
  const int ls = u / a.Hkv;
  r.s = ls % a.b;
  r.l = ls / a.b;
  if (a.varlen) {
    r.tok0 = a.cu_seqlens[r.s];
    r.n = a.cu_seqlens[r.s + 1] - a.cu_seqlens[r.s];
  } else {
    r.tok0 = 0;
    r.n = a.n_max;
  }
  return r;
}

// TMA coordinates (x = element within the token row, y = token row) of token t
// of head `head` in a tensor described by element strides.
struct Coord {
  int32_t x, y;
};

__device__ __forceinline__ Coord tma_coord(int64_t s_layer, int64_t s_seq, int64_t s_head,
                                           int64_t s_tok, bool packed, const Unit& u, int head,
                                           int64_t t) {
  const int64_t base = u.l * s_layer +
                       (packed ? u.tok0 * s_tok : static_cast<int64_t>(u.s) * s_seq) +
                       static_cast<int64_t>(head) * s_head;
  Coord c;
  c.x = static_cast<int32_t>(base % s_tok);
  c.y = static_cast<int32_t>(base / s_tok + t);
  return c;
}

// Row j = g * P + i of a query block is query head g of the group at position
// row_position(); -1 marks rows that do not exist (padding, i >= W_eff, or past
// the sequence end).
__device__ __forceinline__ int row_position(const ScoreArgs& a, int n, int rb, int j) {
  if (j >= a.nrows) return -1;
  const int i = j % a.P;
  if (a.mode == kModeSnapKV) {
    const int w_eff = min(a.W, n);
    return i < w_eff ? n - w_eff + i : -1;
  }
  const int p = rb * a.P + i;
  return p < n ? p : -1;
}

// Smallest position of a query block and whether every one of its rows exists.
__device__ __forceinline__ void row_block_span(const ScoreArgs& a, int n, int rb, int* min_pos,
                                               bool* all_rows) {
  if (a.mode == kModeSnapKV) {
    const int w_eff = min(a.W, n);
    *min_pos = n - w_eff;
    *all_rows = (w_eff == a.W);
  } else {
    *min_pos = rb * a.P;
    *all_rows = (rb + 1) * a.P <= n;
  }
}

// The (key tile, query block) pairs of one CTA, visited as
// for kt in [kt0, kt1): for rb in [rb0, rb1).  Either the key range or the
// query-block range has a single element:
//   pass 1, both scores: one query block, the key tiles of a chunk;
//   pass 2, SnapKV:      one query block (the window), the key tiles of a chunk;
//   pass 2, H2O:         one key tile, every query block at or after it.
struct Work {
  Unit unit;
  int u;
  int kt0, kt1;
  int rb0, rb1;
  int chunk;
};

__device__ __forceinline__ Work decode_work(const ScoreArgs& a, int pass) {
  Work w;
  const int bid = blockIdx.x;
  w.u = bid % a.n_units;
  const int slot = bid / a.n_units;
  w.unit = decode_unit(a, w.u);
  const int n = w.unit.n;
  const int ntiles = (n + kTileKeys - 1) / kTileKeys;
  w.chunk = 0;
  if (a.mode == kModeSnapKV) {
    w.chunk = slot;
    w.kt0 = slot * a.chunk_tiles;
    w.kt1 = min(ntiles, w.kt0 + a.chunk_tiles);
    w.rb0 = 0;
    w.rb1 = n > 0 ? 1 : 0;
  } else {
    // H2O, both passes: one query block, the key tiles up to its last
    // position (pass 2 adds its column sums into the scores atomically)
    const int rb = a.nrb_max - 1 - slot;        // longest query blocks first
    w.rb0 = rb;
    w.rb1 = (rb * a.P < n) ? rb + 1 : rb;
    const int kend = min(n, (rb + 1) * a.P);
    w.kt0 = 0;
    w.kt1 = (kend + kTileKeys - 1) / kTileKeys;
  }
  if (w.kt1 <= w.kt0 || w.rb1 <= w.rb0) {
    w.kt1 = w.kt0;
    w.rb1 = w.rb0;
  }
  return w;
}

__device__ __forceinline__ int64_t score_base(const ScoreArgs& a, const Unit& un, int u) {
  if (a.varlen) return (static_cast<int64_t>(un.l) * a.Hkv + un.h) * a.T + un.tok0;
  return static_cast<int64_t>(u) * a.n_max;
}

// ---------------------------------------------------------------- epilogue --

// NCOL accumulator columns of the calling thread's TMEM lane, as raw bits.
// One wait for all loads; the fence keeps their uses below the wait.
template <int NCOL>
__device__ __forceinline__ void tmem_load_cols(uint32_t taddr, uint32_t* r) {
  __syncwarp();
#pragma unroll
  for (int c = 0; c < NCOL / 32; ++c) tmem_ld32(taddr + c * 32, r + c * 32);
  tmem_wait_ld();
#pragma unroll
  for (int c = 0; c < NCOL / 32; ++c) tmem_reg_fence(r + c * 32);
}

__device__ __forceinline__ float2 bits2(const uint32_t* r, int i) {
  return make_float2(__uint_as_float(r[i]), __uint_as_float(r[i + 1]));
}

__device__ __forceinline__ float2 exp2x2(float2 v) {
  return make_float2(fast_exp2(v.x), fast_exp2(v.y));
}

// sum_i exp2(v_i * c - m): packed f32x2 FMA/ADD, four independent partial sums.
template <int NCOL>
__device__ __forceinline__ float sum_exp2_shift(const uint32_t* r, float c, float m) {
  const float2 cc = make_float2(c, c), mm = make_float2(-m, -m);
  float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                   make_float2(0.f, 0.f)};
#pragma unroll
  for (int i = 0; i < NCOL; i += 8) {
#pragma unroll
    for (int k = 0; k < 4; ++k)
      acc[k] = __fadd2_rn(acc[k], exp2x2(__ffma2_rn(bits2(r, i + 2 * k), cc, mm)));
  }
  const float2 s = __fadd2_rn(__fadd2_rn(acc[0], acc[1]), __fadd2_rn(acc[2], acc[3]));
  return s.x + s.y;
}

__device__ __forceinline__ float max3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

template <int NCOL>
__device__ __forceinline__ float max_cols(const uint32_t* r) {
  float m[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) m[k] = __uint_as_float(r[k]);
#pragma unroll
  for (int i = 4; i + 8 <= NCOL; i += 8)
#pragma unroll
    for (int k = 0; k < 4; ++k)
      m[k] = max3f(m[k], __uint_as_float(r[i + 2 * k]), __uint_as_float(r[i + 2 * k + 1]));
  // the last 4 columns
#pragma unroll
  for (int k = 0; k < 4; ++k) m[k] = fmaxf(m[k], __uint_as_float(r[NCOL - 4 + k]));
  return fmaxf(fmaxf(m[0], m[1]), fmaxf(m[2], m[3]));
}

// One tile of pass 1 for the row at position `pos`: keys t0 .. t0+NCOL-1 with
// raw logits r.  (m2, l) is the running reference and sum of exp2 relative
// to it.  When the tile is fully visible and a reference exists, the tile is
// summed against the current reference; a sum that is non-finite or above
// 1e18 (a much larger logit arrived) is redone with the tile's exact max.
template <int NCOL>
__device__ __forceinline__ void rowstats_tile(const uint32_t* r, int t0, int pos, float c1,
                                              float& m2, float& l) {
  if (pos < 0 || t0 > pos) return;
  const bool whole = (t0 + NCOL - 1 <= pos);
  if (whole && m2 > -INFINITY) {
    const float s = sum_exp2_shift<NCOL>(r, c1, m2);
    if (s <= 1.0e18f) {
      l += s;
      return;
    }
  }
  float mx, s;
  if (whole) {
    mx = max_cols<NCOL>(r) * c1;
    const float mnew = fmaxf(m2, mx);
    s = sum_exp2_shift<NCOL>(r, c1, mnew);
    l = l * fast_exp2(m2 - mnew) + s;
    m2 = mnew;
  } else {
    mx = -INFINITY;
#pragma unroll
    for (int i = 0; i < NCOL; ++i)
      if (t0 + i <= pos) mx = fmaxf(mx, __uint_as_float(r[i]));
    const float mnew = fmaxf(m2, mx * c1);
    s = 0.f;
#pragma unroll
    for (int i = 0; i < NCOL; ++i) {
      const float e = fast_exp2(fmaf(__uint_as_float(r[i]), c1, -mnew));
      s += (t0 + i <= pos) ? e : 0.f;
    }
    l = l * fast_exp2(m2 - mnew) + s;
    m2 = mnew;
  }
}

// One NCOL-key slice of pass 1 for the row at `pos` (keys t0 .. t0+NCOL-1,
// raw logits r, overwritten at the causal edge); (m2, l) as in
// rowstats_tile.  Keys past the row's own position become -inf, so every
// slice takes the same branch-free path: the reference moves to the slice's
// maximum first (three-input max on the ALU), then one packed sum against it.
template <int NCOL>
__device__ __forceinline__ void rowstats_slice(uint32_t* r, int t0, int pos, float c1,
                                               float& m2, float& l) {
  if (pos < 0 || t0 > pos) return;
  if (t0 + NCOL - 1 > pos) {
    const int last = pos - t0;
#pragma unroll
    for (int i = 0; i < NCOL; ++i)
      if (i > last) r[i] = 0xFF800000u;          // -inf
  }
  const float mnew = fmaxf(m2, max_cols<NCOL>(r) * c1);
  const float s = sum_exp2_shift<NCOL>(r, c1, mnew);
  l = l * fast_exp2(m2 - mnew) + s;
  m2 = mnew;
}

// Pass 1 epilogue: the thread owns one query row and NCOL keys of every tile.
// With two row tiles, two parts share each tile (NCOL = 64 keys each); with
// one, all four parts share it (NCOL = 32).  The parts merge at the end.
template <int NCOL>
__device__ __forceinline__ void rowstats_epilogue(const ScoreArgs& a, const Work& w, Shared& sh,
                                                  uint32_t tmem, int n, int warp, int lane,
                                                  int nrt) {
  const int qd = warp & 3;
  const int part = warp >> 2;
  const int rt = (nrt == 2) ? part >> 1 : 0;
  const int sub = (nrt == 2) ? part & 1 : part;
  const int row = rt * 128 + qd * 32 + lane;
  const int col0 = rt * 128 + sub * NCOL;
  const int key0 = sub * NCOL;
  const uint32_t lane_base = static_cast<uint32_t>(qd * 32) << 16;
  const int rb = w.rb0;
  const int pos = (w.rb1 > w.rb0) ? row_position(a, n, rb, row) : -1;
  float m2 = -INFINITY, l = 0.f;
  bool ok = true;
  int pair = 0;
  for (int kt = w.kt0; kt < w.kt1; ++kt) {
    const int ab = pair & 1;
    ok = __all_sync(0xffffffffu, mbar_wait(&sh.acc_full[ab], (pair >> 1) & 1, sh.abort_flag, a.status));
    if (!ok) break;
    tc_fence_after();
    // 32 columns at a time keeps the live registers within the launch bound;
    // the accumulator is released once its last columns are in registers.
    uint32_t r[32];
#pragma unroll
    for (int h = 0; h < NCOL / 32; ++h) {
      tmem_load_cols<32>(tmem + lane_base + ab * 256 + col0 + h * 32, r);
      if (h + 1 == NCOL / 32) {
        tc_fence_before();
        mbar_arrive(&sh.acc_empty[ab]);
      }
      rowstats_tile<32>(r, kt * kTileKeys + key0 + h * 32, pos, a.c1, m2, l);
    }
    ++pair;
  }
  if (!ok) return;
  const int nsub = kParts / nrt;            // parts sharing one row
  if (sub != 0) {
    sh.merge[sub * kRowsMax + row] = make_float2(m2, l);
    mbar_arrive(sh.red_full);
    return;
  }
  if (!mbar_wait(sh.red_full, 0, sh.abort_flag, a.status)) return;
  for (int x = 1; x < nsub; ++x) {
    const float2 o = sh.merge[x * kRowsMax + row];
    const float mm = fmaxf(m2, o.x);
    if (mm > -INFINITY) {
      l = l * fast_exp2(m2 - mm) + o.y * fast_exp2(o.x - mm);
      m2 = mm;
    }
  }
  if (a.mode == kModeSnapKV) {
    const int64_t slot = static_cast<int64_t>(w.u) * a.n_chunks + w.chunk;
    if (in_bounds(slot * kRowsMax + row, 1, a.ext_partials, a.status))
      a.partials[slot * kRowsMax + row] = make_float2(m2, l);
    if (nrt == 1 && in_bounds(slot * kRowsMax + 128 + row, 1, a.ext_partials, a.status))
      a.partials[slot * kRowsMax + 128 + row] = make_float2(-INFINITY, 0.f);
  } else if (w.rb1 > w.rb0) {
    const int64_t o = (static_cast<int64_t>(w.u) * a.nrb_max + rb) * kRowsMax;
    if (in_bounds(o + row, 1, a.ext_lse2, a.status))
      a.lse2[o + row] = (l > 0.f) ? -(m2 + __log2f(l)) : -INFINITY;
    if (nrt == 1 && in_bounds(o + 128 + row, 1, a.ext_lse2, a.status)) a.lse2[o + 128 + row] = -INFINITY;
  }
}

// Pass 2 epilogue: the thread owns key lane `kl` of the tile and NCOL query
// rows (one quarter of the block); the parts add up at the end of each tile.
// sh.lse holds the negated log2 normalisers (-inf for rows that do not exist).
template <int SQ, int NCOL>
__device__ __forceinline__ void colsum_epilogue(const ScoreArgs& a, const Work& w, Shared& sh,
                                                uint32_t tmem, int n, int warp, int lane,
                                                bool q_streams) {
  const int qd = warp & 3;
  const int part = warp >> 2;
  const uint32_t lane_base = static_cast<uint32_t>(qd * 32) << 16;
  const int kl = qd * 32 + lane;
  const int j0 = part * NCOL;
  const int64_t sbase = score_base(a, w.unit, w.u);
  const float c1 = a.c1;
  const float2 cc = make_float2(c1, c1);
  bool ok = true;
  int pair = 0, quse = 0, xchg = 0;
  for (int kt = w.kt0; kt < w.kt1 && ok; ++kt) {
    const int t = kt * kTileKeys + kl;
    float colsum = 0.f;
    for (int rb = w.rb0; rb < w.rb1; ++rb) {
      if (q_streams || kt == w.kt0) {
        // Acquire the producer's normalisers and positions for this block.
        ok = __all_sync(0xffffffffu, mbar_wait(&sh.q_full[quse % SQ], (quse / SQ) & 1,
                                               sh.abort_flag, a.status));
        if (!ok) break;
        ++quse;
      }
      const int qslot = (quse - 1) % SQ;
      int min_pos;
      bool all_rows;
      row_block_span(a, n, rb, &min_pos, &all_rows);
      const bool fast = all_rows && (kt * kTileKeys + kTileKeys - 1 <= min_pos);
      const int ab = pair & 1;
      ok = __all_sync(0xffffffffu, mbar_wait(&sh.acc_full[ab], (pair >> 1) & 1, sh.abort_flag, a.status));
      if (!ok) break;
      tc_fence_after();
      uint32_t r[NCOL];
      tmem_load_cols<NCOL>(tmem + lane_base + ab * 256 + j0, r);
      tc_fence_before();
      mbar_arrive(&sh.acc_empty[ab]);
      const float* nl = sh.lse + qslot * kRowsMax + j0;
      if (fast) {
        float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                         make_float2(0.f, 0.f)};
#pragma unroll
        for (int i = 0; i < NCOL; i += 8) {
          const float4 L0 = *reinterpret_cast<const float4*>(nl + i);
          const float4 L1 = *reinterpret_cast<const float4*>(nl + i + 4);
          acc[0] = __fadd2_rn(acc[0], exp2x2(__ffma2_rn(bits2(r, i), cc, make_float2(L0.x, L0.y))));
          acc[1] = __fadd2_rn(acc[1], exp2x2(__ffma2_rn(bits2(r, i + 2), cc, make_float2(L0.z, L0.w))));
          acc[2] = __fadd2_rn(acc[2], exp2x2(__ffma2_rn(bits2(r, i + 4), cc, make_float2(L1.x, L1.y))));
          acc[3] = __fadd2_rn(acc[3], exp2x2(__ffma2_rn(bits2(r, i + 6), cc, make_float2(L1.z, L1.w))));
        }
        const float2 s2 = __fadd2_rn(__fadd2_rn(acc[0], acc[1]), __fadd2_rn(acc[2], acc[3]));
        colsum += s2.x + s2.y;
      } else {
        float s = 0.f;
#pragma unroll
        for (int i = 0; i < NCOL; ++i) {
          const float e = fast_exp2(fmaf(__uint_as_float(r[i]), c1, nl[i]));
          s += (t <= row_position(a, n, rb, j0 + i)) ? e : 0.f;
        }
        colsum += s;
      }
      if (q_streams || kt + 1 == w.kt1) mbar_arrive(&sh.q_empty[qslot]);
      ++pair;
    }
    if (!ok) break;
    // Add the row parts of this key and write s(t).
    if (part != 0) {
      ok = mbar_wait(sh.red_empty, (xchg & 1) ^ 1, sh.abort_flag, a.status);
      if (!ok) break;
      sh.red[(part - 1) * kTileKeys + kl] = colsum;
      mbar_arrive(sh.red_full);
    } else {
      ok = mbar_wait(sh.red_full, xchg & 1, sh.abort_flag, a.status);
      if (!ok) break;
      float total = colsum;
#pragma unroll
      for (int x = 1; x < kParts; ++x) total += sh.red[(x - 1) * kTileKeys + kl];
      mbar_arrive(sh.red_empty);
      if (t < n && in_bounds(sbase + t, 1, a.ext_scores, a.status)) {
        if (a.mode == kModeH2O)
          atomicAdd(a.prepool + sbase + t, total);   // one query block's share
        else
          a.prepool[sbase + t] = total;
      }
    }
    ++xchg;
  }
}

// ------------------------------------------------------------------ kernel --

template <int D, int PASS>
__global__ void __launch_bounds__(kThreads, 1)
    attn_pass_kernel(const __grid_constant__ CUtensorMap k_map,
                     const __grid_constant__ CUtensorMap q_map, const ScoreArgs a) {
  using C = Cfg<D, PASS>;
  extern __shared__ uint8_t smem_raw[];
  Shared sh = carve<D, PASS>(smem_raw);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  const Work w = decode_work(a, PASS);
  const int nrt = a.nrows_pad / 128;
  const int n = w.unit.n;
  // Every CTA keeps one query block for its whole life and streams key tiles.
  const bool q_streams = false;

  // ---- set-up: barriers, zeroed padding rows, tensor memory
  if (threadIdx.x == 0) {
    for (int i = 0; i < C::SK; ++i) {
      mbar_init(&sh.k_full[i], 1);
      mbar_init(&sh.k_empty[i], 1);
    }
    for (int i = 0; i < C::SQ; ++i) {
      mbar_init(&sh.q_full[i], 1);
      mbar_init(&sh.q_empty[i], PASS == kPassColsum ? 1 + kEpiWarps * 32 : 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sh.acc_full[i], 1);
      mbar_init(&sh.acc_empty[i], kEpiWarps * 32);
    }
    // non-leader parts hand their partial results to the leader part
    mbar_init(sh.red_full, PASS == kPassColsum ? (kParts - 1) * 128 : (kParts - nrt) * 128);
    mbar_init(sh.red_empty, 128);
    mbar_init(sh.drain, 1);
    *sh.abort_flag = 0;
    fence_mbar_init();
  }
  if (a.nrows < a.nrows_pad) {
    // Query rows past the block are never loaded; zero them once so the MMA
    // reads finite values there.
    const int words = (a.nrows_pad - a.nrows) * 32;   // 128 bytes per half-row
    for (int slot = 0; slot < C::SQ; ++slot)
      for (int hf = 0; hf < C::kHalves; ++hf) {
        uint32_t* dst = reinterpret_cast<uint32_t*>(sh.q + slot * C::kQSlotBytes +
                                                    hf * C::kQHalfBytes + a.nrows * 128);
        for (int i = threadIdx.x; i < words; i += kThreads) dst[i] = 0u;
      }
    fence_proxy_async_smem();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(sh.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  if (warp == kProducerWarp && lane == 0) {
    tma_prefetch_map(&k_map);
    tma_prefetch_map(&q_map);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *sh.tmem_base;

  if (warp == kProducerWarp) {
    // ------------------------------------------------------------- producer
    int kload = 0, qload = 0;
    bool ok = true;
    for (int kt = w.kt0; kt < w.kt1 && ok; ++kt) {
      {
        const int slot = kload % C::SK;
        if (lane == 0)
          ok = mbar_wait(&sh.k_empty[slot], ((kload / C::SK) & 1) ^ 1, sh.abort_flag, a.status);
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) break;
        if (lane == 0) {
          mbar_arrive_expect_tx(&sh.k_full[slot], C::kKTileBytes);
          const Coord c = tma_coord(a.k_layer, a.k_seq, a.k_head, a.k_tok, a.varlen != 0, w.unit,
                                    w.unit.h, static_cast<int64_t>(kt) * kTileKeys);
          uint8_t* dst = sh.k + slot * C::kKTileBytes;
#pragma unroll
          for (int hf = 0; hf < C::kHalves; ++hf)
            tma_load_2d(dst + hf * C::kKHalfBytes, &k_map, c.x + hf * 64, c.y, &sh.k_full[slot]);
        }
        ++kload;
      }
      for (int rb = w.rb0; rb < w.rb1; ++rb) {
        if (!q_streams && kt != w.kt0) break;           // the one query block is loaded
        const int slot = qload % C::SQ;
        if (lane == 0)
          ok = mbar_wait(&sh.q_empty[slot], ((qload / C::SQ) & 1) ^ 1, sh.abort_flag, a.status);
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) break;
        if (lane == 0) {
          const uint32_t nl_bytes = (PASS == kPassColsum) ? kRowsMax * 4 : 0;
          mbar_arrive_expect_tx(&sh.q_full[slot], static_cast<uint32_t>(a.nrows) * D * 2 + nl_bytes);
          if (PASS == kPassColsum) {
            // the block's negated normalisers (-inf where a row does not exist)
            const int64_t lrow =
                (static_cast<int64_t>(w.u) * (a.mode == kModeSnapKV ? 1 : a.nrb_max) + rb) * kRowsMax;
            bulk_copy_g2s(sh.lse + slot * kRowsMax, a.lse2 + lrow, nl_bytes, &sh.q_full[slot]);
          }
          uint8_t* dst = sh.q + slot * C::kQSlotBytes;
          const bool window = (a.mode == kModeSnapKV);
          const int64_t t0 = window ? 0 : static_cast<int64_t>(rb) * a.P;
          for (int g = 0; g < a.G; ++g) {
            const Coord c = tma_coord(a.q_layer, a.q_seq, a.q_head, a.q_tok,
                                      !window && a.varlen != 0, w.unit, w.unit.h * a.G + g, t0);
#pragma unroll
            for (int hf = 0; hf < C::kHalves; ++hf)
              tma_load_2d(dst + hf * C::kQHalfBytes + g * a.P * 128, &q_map, c.x + hf * 64, c.y,
                          &sh.q_full[slot]);
          }
        }
        ++qload;
      }
    }
    // After an abort, let copies still in flight land before the CTA exits.
    if (*sh.abort_flag && lane == 0) {
      for (int i = 0; i < min(kload, C::SK); ++i) {
        const int ld = kload - 1 - i;
        mbar_wait(&sh.k_full[ld % C::SK], (ld / C::SK) & 1, nullptr, nullptr);
      }
      for (int i = 0; i < min(qload, C::SQ); ++i) {
        const int ld = qload - 1 - i;
        mbar_wait(&sh.q_full[ld % C::SQ], (ld / C::SQ) & 1, nullptr, nullptr);
      }
    }
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------------ MMA
    int kuse = 0, quse = 0, pair = 0;
    bool ok = true;
    const uint32_t idesc = (PASS == kPassRowstats) ? idesc_bf16_f32(128, kTileKeys)
                                                   : idesc_bf16_f32(128, a.nrows_pad);
    for (int kt = w.kt0; kt < w.kt1 && ok; ++kt) {
      const int kslot = kuse % C::SK;
      if (lane == 0) ok = mbar_wait(&sh.k_full[kslot], (kuse / C::SK) & 1, sh.abort_flag, a.status);
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      for (int rb = w.rb0; rb < w.rb1; ++rb) {
        const bool new_q = q_streams || kt == w.kt0;
        if (new_q) {
          if (lane == 0)
            ok = mbar_wait(&sh.q_full[quse % C::SQ], (quse / C::SQ) & 1, sh.abort_flag, a.status);
          ok = __shfl_sync(0xffffffffu, ok, 0);
          if (!ok) break;
          ++quse;
        }
        const int qslot = (quse - 1) % C::SQ;
        const int ab = pair & 1;
        if (lane == 0)
          ok = mbar_wait(&sh.acc_empty[ab], ((pair >> 1) & 1) ^ 1, sh.abort_flag, a.status);
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) break;
        tc_fence_after();
        if (lane == 0) {
          const uint32_t qbase = smem_u32(sh.q + qslot * C::kQSlotBytes);
          const uint32_t kbase = smem_u32(sh.k + kslot * C::kKTileBytes);
          const uint32_t dcol = tmem + ab * 256;
          if (PASS == kPassRowstats) {
            for (int rt = 0; rt < nrt; ++rt) {
#pragma unroll
              for (int ks = 0; ks < C::kKSteps; ++ks) {
                const uint32_t koff = (ks & 3) * 32;
                const uint64_t ad = sdesc_kmajor_sw128(qbase + (ks >> 2) * C::kQHalfBytes +
                                                       rt * 128 * 128 + koff);
                const uint64_t bd = sdesc_kmajor_sw128(kbase + (ks >> 2) * C::kKHalfBytes + koff);
                mma_bf16_ss(dcol + rt * kTileKeys, ad, bd, idesc, ks > 0 ? 1u : 0u);
              }
            }
          } else {
#pragma unroll
            for (int ks = 0; ks < C::kKSteps; ++ks) {
              const uint32_t koff = (ks & 3) * 32;
              const uint64_t ad = sdesc_kmajor_sw128(kbase + (ks >> 2) * C::kKHalfBytes + koff);
              const uint64_t bd = sdesc_kmajor_sw128(qbase + (ks >> 2) * C::kQHalfBytes + koff);
              mma_bf16_ss(dcol, ad, bd, idesc, ks > 0 ? 1u : 0u);
            }
          }
          mma_commit(&sh.acc_full[ab]);
          // A query block is released after its last pair, a key tile after
          // the last query block paired with it.
          const bool q_last = q_streams || (kt + 1 == w.kt1);
          if (q_last) mma_commit(&sh.q_empty[qslot]);
          if (rb + 1 == w.rb1) mma_commit(&sh.k_empty[kslot]);
        }
        __syncwarp();
        ++pair;
      }
      ++kuse;
    }
    // No MMA may still be writing tensor memory when it is freed.
    if (lane == 0) {
      mma_commit(sh.drain);
      mbar_wait(sh.drain, 0, nullptr, nullptr);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------- epilogue
    if (PASS == kPassRowstats) {
      if (nrt == 2)
        rowstats_epilogue<64>(a, w, sh, tmem, n, warp, lane, nrt);
      else
        rowstats_epilogue<32>(a, w, sh, tmem, n, warp, lane, nrt);
    } else {
      if (a.nrows_pad == 256)
        colsum_epilogue<C::SQ, 64>(a, w, sh, tmem, n, warp, lane, q_streams);
      else
        colsum_epilogue<C::SQ, 32>(a, w, sh, tmem, n, warp, lane, q_streams);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------- fused SnapKV / H2O score --

template <int D>
struct FCfg {
  static constexpr int kHalves = D / 64;
  static constexpr int kKSteps = D / 16;
  static constexpr int kKTileBytes = kTileKeys * D * 2;
  static constexpr int kQSlotBytes = kRowsMax * D * 2;
  static constexpr int kKHalfBytes = kTileKeys * 128;
  static constexpr int kQHalfBytes = kRowsMax * 128;
  static constexpr int SK = 4;
  static constexpr int kQOff = 0;
  static constexpr int kKOff = kQOff + kQSlotBytes;
  static constexpr int kPosOff = kKOff + SK * kKTileBytes;
  static constexpr int kRedOff = kPosOff + kRowsMax * 4;
  static constexpr int kMergeOff = kRedOff + (kParts - 1) * kTileKeys * 4;
  // the extra pass-2 k-step: row normalisers (256 rows) against ones (128
  // keys), 16 bf16 columns each, K-major without swizzle
  static constexpr int kNlOff = kMergeOff + kParts * kRowsMax * 8;
  static constexpr int kOnesOff = kNlOff + kRowsMax * 32;
  static constexpr int kBarOff = kOnesOff + kTileKeys * 32;
  // k_full/k_empty[SK], q_full, q_empty, acc_full[2], acc_empty[2], merge_full,
  // red_full[2], red_empty[2], drain, pub, lse_go, lse_ready
  static constexpr int kNumBars = 2 * SK + 15;
  static constexpr int kMiscOff = kBarOff + kNumBars * 8;
  static constexpr int kBytes = kMiscOff + 32;
  static constexpr int kSmemAlloc = kBytes + 1024;
};

struct FShared {
  uint8_t* q;
  uint8_t* k;
  uint8_t* nlb;      // [256 rows][16] bf16: -lse2_j / c1 in three parts, then zeros
  uint8_t* ones;     // [128 keys][16] bf16: 1, 1, 1, then zeros
  int32_t* pos;
  float* red;
  float2* merge;
  uint64_t *k_full, *k_empty, *q_full, *q_empty, *acc_full, *acc_empty;
  uint64_t *merge_full, *red_full, *red_empty, *drain;
  uint64_t *pub, *lse_go, *lse_ready;
  uint32_t* tmem_base;
  volatile int* abort_flag;
};

template <int D>
__device__ __forceinline__ FShared fcarve(uint8_t* raw) {
  using C = FCfg<D>;
  const uint32_t a = smem_u32(raw);
  uint8_t* base = raw + ((1024u - (a & 1023u)) & 1023u);
  FShared s;
  s.q = base + C::kQOff;
  s.k = base + C::kKOff;
  s.pos = reinterpret_cast<int32_t*>(base + C::kPosOff);
  s.red = reinterpret_cast<float*>(base + C::kRedOff);
  s.merge = reinterpret_cast<float2*>(base + C::kMergeOff);
  s.nlb = base + C::kNlOff;
  s.ones = base + C::kOnesOff;
  uint64_t* b = reinterpret_cast<uint64_t*>(base + C::kBarOff);
  s.k_full = b;
  s.k_empty = b + C::SK;
  b += 2 * C::SK;
  s.q_full = b++;
  s.q_empty = b++;
  s.acc_full = b;
  b += 2;
  s.acc_empty = b;
  b += 2;
  s.merge_full = b++;
  s.red_full = b;
  b += 2;
  s.red_empty = b;
  b += 2;
  s.drain = b++;
  s.pub = b++;
  s.lse_go = b++;
  s.lse_ready = b++;
  s.tmem_base = reinterpret_cast<uint32_t*>(base + C::kMiscOff);
  s.abort_flag = reinterpret_cast<volatile int*>(base + C::kMiscOff + 4);
  return s;
}

// Element index (in bf16 units) of (row r, column kk < 16) in a K-major block
// of 16 columns without swizzle: 8-row x 8-column core matrices of 128 bytes,
// the two column halves 128 bytes apart, 8-row groups 256 bytes apart.
__device__ __forceinline__ int nl_elem(int r, int kk) {
  return ((r >> 3) * 256 + (kk >> 3) * 128 + (r & 7) * 16 + (kk & 7) * 2) >> 1;
}

__device__ __forceinline__ uint16_t bf16_bits_rn(float x) {
  return __bfloat16_as_ushort(__float2bfloat16_rn(x));
}

__device__ __forceinline__ float bf16_value(uint16_t b) {
  return __uint_as_float(static_cast<uint32_t>(b) << 16);
}

__device__ __forceinline__ int ld_acquire_gpu(const int32_t* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Key-tile range of chunk c of a unit with n keys: the unit's tiles split as
// evenly as possible over its n_chunks chunks (sequences of a varlen batch
// keep their whole gang busy).
__device__ __forceinline__ void chunk_tiles(const ScoreArgs& a, int n, int c, int* kt0, int* kt1) {
  const int ntiles = (n + kTileKeys - 1) / kTileKeys;
  const int ct = (ntiles + a.n_chunks - 1) / a.n_chunks;
  *kt0 = min(ntiles, c * ct);
  *kt1 = min(ntiles, *kt0 + ct);
}

// Item `item` of the fused launch.  SnapKV: (unit, chunk of its key tiles).
// H2O: (unit, query block), the longest blocks first, over the key tiles up
// to the block's last position; its rows' normalisers are its own (no other
// CTA contributes), so the block needs no cross-CTA exchange.
struct FItem {
  int u, chunk, rb, kt0, kt1;
  Unit un;
};

__device__ __forceinline__ FItem fused_item(const ScoreArgs& a, int item) {
  FItem it;
  if (a.mode == kModeSnapKV) {
    it.u = item / a.n_chunks;
    it.chunk = item % a.n_chunks;
    it.rb = 0;
    it.un = decode_unit(a, it.u);
    chunk_tiles(a, it.un.n, it.chunk, &it.kt0, &it.kt1);
  } else {
    it.u = item % a.n_units;
    it.chunk = 0;
    it.rb = a.nrb_max - 1 - item / a.n_units;
    it.un = decode_unit(a, it.u);
    const int n = it.un.n;
    it.kt0 = 0;
    it.kt1 = (it.rb * a.P < n) ? (min(n, (it.rb + 1) * a.P) + kTileKeys - 1) / kTileKeys : 0;
  }
  return it;
}

// Descriptor `d` moved `bytes` further into shared memory.  The start-address
// field is the low 14 bits (16-byte units) and every operand stays inside
// shared memory, so the add never carries out of the low word.
__device__ __forceinline__ uint64_t desc_plus(uint64_t d, uint32_t bytes) {
  const uint32_t lo = static_cast<uint32_t>(d) + (bytes >> 4);
  return (d & 0xFFFFFFFF00000000ull) | lo;
}

template <int D>
__device__ __forceinline__ void issue_mma_rows_on_lanes(uint64_t dq, uint64_t dk,
                                                        uint32_t dcol, int nrt) {
  using C = FCfg<D>;
  const uint32_t idesc = idesc_bf16_f32(128, kTileKeys);
  for (int rt = 0; rt < nrt; ++rt) {
    const uint64_t dqr = desc_plus(dq, rt * 128 * 128);
#pragma unroll
    for (int ks = 0; ks < C::kKSteps; ++ks) {
      const uint32_t koff = (ks & 3) * 32;
      const uint64_t ad = desc_plus(dqr, (ks >> 2) * C::kQHalfBytes + koff);
      const uint64_t bd = desc_plus(dk, (ks >> 2) * C::kKHalfBytes + koff);
      mma_bf16_ss(dcol + rt * kTileKeys, ad, bd, idesc, ks > 0 ? 1u : 0u);
    }
  }
}

template <int D>
__device__ __forceinline__ void issue_mma_keys_on_lanes(uint64_t dq, uint64_t dk,
                                                        uint32_t dcol, int nrows_pad) {
  using C = FCfg<D>;
  const uint32_t idesc = idesc_bf16_f32(128, nrows_pad);
#pragma unroll
  for (int ks = 0; ks < C::kKSteps; ++ks) {
    const uint32_t koff = (ks & 3) * 32;
    const uint64_t ad = desc_plus(dk, (ks >> 2) * C::kKHalfBytes + koff);
    const uint64_t bd = desc_plus(dq, (ks >> 2) * C::kQHalfBytes + koff);
    mma_bf16_ss(dcol, ad, bd, idesc, ks > 0 ? 1u : 0u);
  }
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    snapkv_fused_kernel(const __grid_constant__ CUtensorMap k_map,
                        const __grid_constant__ CUtensorMap q_map, const FusedArgs fa) {
  using C = FCfg<D>;
  const ScoreArgs& a = fa.s;
  extern __shared__ uint8_t smem_raw[];
  FShared sh = fcarve<D>(smem_raw);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int nrt = a.nrows_pad / 128;

  if (threadIdx.x == 0) {
    for (int i = 0; i < C::SK; ++i) {
      mbar_init(&sh.k_full[i], 1);
      mbar_init(&sh.k_empty[i], 1);
    }
    mbar_init(sh.q_full, 1);
    mbar_init(sh.q_empty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sh.acc_full[i], 1);
      mbar_init(&sh.acc_empty[i], (kEpiWarps / 2) * 32);   // one group per buffer
      mbar_init(&sh.red_full[i], 128);
      mbar_init(&sh.red_empty[i], 128);
    }
    mbar_init(sh.merge_full, (kParts - nrt) * 128);
    mbar_init(sh.drain, 1);
    mbar_init(sh.pub, kEpiWarps * 32);
    mbar_init(sh.lse_go, 1);
    mbar_init(sh.lse_ready, kEpiWarps * 32);
    *sh.abort_flag = 0;
    fence_mbar_init();
  }
  if (a.nrows < a.nrows_pad) {
    const int words = (a.nrows_pad - a.nrows) * 32;
    for (int hf = 0; hf < C::kHalves; ++hf) {
      uint32_t* dst = reinterpret_cast<uint32_t*>(sh.q + hf * C::kQHalfBytes + a.nrows * 128);
      for (int i = threadIdx.x; i < words; i += kThreads) dst[i] = 0u;
    }
  }
  // Operands of the extra pass-2 k-step, which adds each row's normaliser to
  // its logits in the accumulator: keys x [1, 1, 1, 0 ...] against rows x
  // [three bf16 parts of -lse2_j / c1, 0 ...] (the parts are written per item).
  for (int i = threadIdx.x; i < kTileKeys * 16; i += kThreads) {
    const int r = i >> 4, kk = i & 15;
    reinterpret_cast<uint16_t*>(sh.ones)[nl_elem(r, kk)] = kk < 3 ? 0x3F80u : 0u;   // bf16 1.0
  }
  for (int i = threadIdx.x; i < kRowsMax * 8; i += kThreads) reinterpret_cast<uint32_t*>(sh.nlb)[i] = 0u;
  fence_proxy_async_smem();
  if (warp == kMmaWarp) {
    tmem_alloc(sh.tmem_base, kTmemCols);
    tmem_relinquish();
  }
  if (warp == kProducerWarp && lane == 0) {
    tma_prefetch_map(&k_map);
    tma_prefetch_map(&q_map);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *sh.tmem_base;

  if (warp == kProducerWarp) {
    // ------------------------------------------------------------- producer
    if (lane == 0) {
      // Pass-1 tiles and the window queries are read again soon (pass 2, the
      // unit's other chunks): keep them in L2; pass-2 reads are their last.
      const uint64_t keep = l2_policy_evict_last();
      const uint64_t drop = l2_policy_evict_first();
      int kload = 0, qload = 0;
      // Items are dealt round-robin: the grid is a multiple of the chunks per
      // unit, so a unit's chunks run on different CTAs in the same round.
      const bool h2o = a.mode == kModeH2O;
      for (int item = blockIdx.x; item < fa.n_items; item += gridDim.x) {
        const FItem it = fused_item(a, item);
        const Unit& un = it.un;
        const int kt0 = it.kt0, kt1 = it.kt1;
        if (kt1 == kt0) continue;
        // the item's query rows: the unit's window (SnapKV) or query block (H2O)
        if (!mbar_wait(sh.q_empty, (qload & 1) ^ 1, sh.abort_flag, a.status)) break;
        mbar_arrive_expect_tx(sh.q_full, static_cast<uint32_t>(a.nrows) * D * 2);
        for (int g = 0; g < a.G; ++g) {
          const Coord c = tma_coord(a.q_layer, a.q_seq, a.q_head, a.q_tok, h2o && a.varlen != 0, un,
                                    un.h * a.G + g, h2o ? static_cast<int64_t>(it.rb) * a.P : 0);
#pragma unroll
          for (int hf = 0; hf < C::kHalves; ++hf)
            tma_load_2d_hint(sh.q + hf * C::kQHalfBytes + g * a.P * 128, &q_map, c.x + hf * 64,
                             c.y, sh.q_full, keep);
        }
        ++qload;
        // the chunk's key tiles, once for each pass
        bool ok = true;
        for (int pass = fa.single; pass < 2 && ok; ++pass)
          for (int kt = kt0; kt < kt1; ++kt) {
            const int slot = kload % C::SK;
            if (!mbar_wait(&sh.k_empty[slot], ((kload / C::SK) & 1) ^ 1, sh.abort_flag, a.status)) {
              ok = false;
              break;
            }
            mbar_arrive_expect_tx(&sh.k_full[slot], C::kKTileBytes);
            const Coord c = tma_coord(a.k_layer, a.k_seq, a.k_head, a.k_tok, a.varlen != 0, un,
                                      un.h, static_cast<int64_t>(kt) * kTileKeys);
#pragma unroll
            for (int hf = 0; hf < C::kHalves; ++hf)
              tma_load_2d_hint(sh.k + slot * C::kKTileBytes + hf * C::kKHalfBytes, &k_map,
                               c.x + hf * 64, c.y, &sh.k_full[slot], pass == 0 ? keep : drop);
            ++kload;
          }
        if (!ok) break;
      }
      if (*sh.abort_flag) {
        for (int i = 0; i < min(kload, C::SK); ++i) {
          const int ld = kload - 1 - i;
          mbar_wait(&sh.k_full[ld % C::SK], (ld / C::SK) & 1, nullptr, nullptr);
        }
        if (qload > 0) mbar_wait(sh.q_full, (qload - 1) & 1, nullptr, nullptr);
      }
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------------------ MMA
    if (lane == 0) {
      int kuse = 0, quse = 0, pair = 0;
      int lpop = 0;                                // items whose normalisers the epilogue forms
      bool ok = true;
      const uint64_t ones_desc = sdesc_kmajor_noswizzle(smem_u32(sh.ones), 128, 256);
      const uint64_t nl_desc = sdesc_kmajor_noswizzle(smem_u32(sh.nlb), 128, 256);
      // pass 2 spans only the rows that exist, rounded up to 32 (224 of 256 at G = 7)
      const int p2n = a.nrows_pad == 256 ? ((a.nrows + 31) & ~31) : a.nrows_pad;
      const uint32_t idesc_nl = idesc_bf16_f32(128, p2n);
      for (int item = blockIdx.x; item < fa.n_items && ok; item += gridDim.x) {
        const FItem it = fused_item(a, item);
        const int kt0 = it.kt0, kt1 = it.kt1;
        if (kt1 == kt0) {
          if (a.mode != kModeH2O) ++lpop;          // (the epilogue still forms them)
          continue;
        }
        if (!mbar_wait(sh.q_full, quse & 1, sh.abort_flag, a.status)) break;
        ++quse;
        const uint64_t dq = sdesc_kmajor_sw128(smem_u32(sh.q));
        bool nl_ready = false;
        for (int pass = fa.single; pass < 2 && ok; ++pass)
          for (int kt = kt0; kt < kt1; ++kt) {
            const int kslot = kuse % C::SK;
            const int ab = pair & 1;
            if (!mbar_wait(&sh.k_full[kslot], (kuse / C::SK) & 1, sh.abort_flag, a.status) ||
                !mbar_wait(&sh.acc_empty[ab], ((pair >> 1) & 1) ^ 1, sh.abort_flag, a.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint64_t dk = sdesc_kmajor_sw128(smem_u32(sh.k + kslot * C::kKTileBytes));
            if (pass == 0) {
              issue_mma_rows_on_lanes<D>(dq, dk, tmem + ab * 256, nrt);
            } else {
              issue_mma_keys_on_lanes<D>(dq, dk, tmem + ab * 256, p2n);
              // add the rows' normalisers (once the epilogue has written them)
              if (!nl_ready) {
                if (!mbar_wait(sh.lse_ready, lpop & 1, sh.abort_flag, a.status)) {
                  ok = false;
                  break;
                }
                nl_ready = true;
              }
              mma_bf16_ss(tmem + ab * 256, ones_desc, nl_desc, idesc_nl, 1u);
            }
            mma_commit(&sh.acc_full[ab]);
            mma_commit(&sh.k_empty[kslot]);
            ++kuse;
            ++pair;
          }
        if (ok) mma_commit(sh.q_empty);
        ++lpop;
      }
      mma_commit(sh.drain);
      mbar_wait(sh.drain, 0, nullptr, nullptr);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------- epilogue
    // Two groups of eight warps own the two accumulator buffers (group g the
    // tiles with pair parity g): while one group computes on its tile the
    // other drains the next one from tensor memory.
    const int grp = warp >> 3;
    const int gw = warp & 7;
    const int qd = gw & 3;
    const int gp = gw >> 2;                        // part within the group
    const uint32_t lane_base = static_cast<uint32_t>(qd * 32) << 16;
    const int etid = threadIdx.x;                  // 0 .. kEpiWarps*32-1
    // pass 1 mapping: one query row and all keys of each owned tile (two row
    // tiles) or half of them (one row tile); the row's partial sums from the
    // other group / part merge at the end of the chunk
    const int rt = (nrt == 2) ? gp : 0;
    const int sub = (nrt == 2) ? grp : grp * 2 + gp;
    const int row = rt * 128 + qd * 32 + lane;
    const int p1cols = (nrt == 2) ? 128 : 64;
    const int col1 = rt * 128 + ((nrt == 2) ? 0 : gp * 64);
    const int key1 = (nrt == 2) ? 0 : gp * 64;
    const int nsub = kParts / nrt;
    // pass 2 mapping: one key lane, half of the rows of each owned tile
    const int kl = qd * 32 + lane;
    // (with two row tiles the second part takes the rows past 128 that exist,
    // rounded up to 32, as pass 2's MMA computes only those)
    const int p2cols = a.nrows_pad == 128 ? 64 : (gp == 0 ? 128 : ((a.nrows + 31) & ~31) - 128);
    const int j0 = a.nrows_pad == 128 ? gp * 64 : gp * 128;
    const float c1 = a.c1;
    const float2 cc = make_float2(c1, c1);
    int pair = 0, xchg = 0;
    bool ok = true;
    int ipop = 0;                                  // items done: barrier phases
    const bool h2o = a.mode == kModeH2O;
    for (int item = blockIdx.x; item < fa.n_items && ok; item += gridDim.x) {
      const FItem it = fused_item(a, item);
      const int u = it.u, chunk = it.chunk, rb = it.rb;
      const Unit& un = it.un;
      const int n = un.n;
      const int kt0 = it.kt0, kt1 = it.kt1;
      if (h2o && kt1 == kt0) continue;           // a block past its sequence's end

      if (!fa.single) {
      // ---- pass 1: running (max2, sum) of this thread's row over its keys
      const int pos = row_position(a, n, rb, row);
      float m2 = -INFINITY, l = 0.f;
      for (int kt = kt0; kt < kt1; ++kt, ++pair) {
        const int ab = pair & 1;
        if (ab != grp) continue;                   // the other group's tile
        ok = __all_sync(0xffffffffu, mbar_wait(&sh.acc_full[ab], (pair >> 1) & 1, sh.abort_flag, a.status));
        if (!ok) break;
        tc_fence_after();
        uint32_t r[64];
        for (int h = 0; h < p1cols / 64; ++h) {
          tmem_load_cols<64>(tmem + lane_base + ab * 256 + col1 + h * 64, r);
          if (h + 1 == p1cols / 64) {
            tc_fence_before();
            mbar_arrive(&sh.acc_empty[ab]);
          }
          rowstats_slice<64>(r, kt * kTileKeys + key1 + h * 64, pos, c1, m2, l);
        }
      }
      if (!ok) break;
      // merge the key slices of each row, publish the chunk's partials
      if (sub != 0) {
        sh.merge[sub * kRowsMax + row] = make_float2(m2, l);
        mbar_arrive(sh.merge_full);
      } else {
        ok = mbar_wait(sh.merge_full, ipop & 1, sh.abort_flag, a.status);
        for (int x = 1; x < nsub && ok; ++x) {
          const float2 o = sh.merge[x * kRowsMax + row];
          const float mm = fmaxf(m2, o.x);
          if (mm > -INFINITY) {
            l = l * fast_exp2(m2 - mm) + o.y * fast_exp2(o.x - mm);
            m2 = mm;
          }
        }
        if (h2o) {
          sh.merge[row] = make_float2(m2, l);      // (slot 0: the leader's own)
        } else {
          const int64_t slot = static_cast<int64_t>(u) * a.n_chunks + chunk;
          if (in_bounds(slot * kRowsMax + row, 1, a.ext_partials, a.status))
            a.partials[slot * kRowsMax + row] = make_float2(m2, l);
          if (nrt == 1 && in_bounds(slot * kRowsMax + 128 + row, 1, a.ext_partials, a.status))
            a.partials[slot * kRowsMax + 128 + row] = make_float2(-INFINITY, 0.f);
          __threadfence();
        }
      }
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) break;
      mbar_arrive(sh.pub);
      if (etid == 0) {
        // every row of this chunk is visible: count it, then wait for the
        // unit's other chunks (bounded)
        bool got = mbar_wait(sh.pub, ipop & 1, sh.abort_flag, a.status);
        if (got && !h2o) {
          __threadfence();
          atomicAdd(fa.work + 1 + u, 1);
          const uint64_t t0 = global_timer_ns();
          while (ld_acquire_gpu(fa.work + 1 + u) < a.n_chunks + fa.hold) {
            if (*sh.abort_flag || global_timer_ns() - t0 > fa.wait_ns) {
              *sh.abort_flag = 1;
              if (a.status) atomicOr(a.status, ROLEKV_STATUS_TIMEOUT);
              got = false;
              break;
            }
            __nanosleep(128);
          }
        }
        mbar_arrive(sh.lse_go);
      }
      ok = __all_sync(0xffffffffu, mbar_wait(sh.lse_go, ipop & 1, sh.abort_flag, a.status));
      if (!ok || *sh.abort_flag) break;
      }  // pass 1
      // ---- normalisers of the unit's rows from all chunks' partials (or,
      // with caller-supplied window normalisers, as snapkv_lse_kernel wrote them)
      if (etid < kRowsMax) {
        const int j = etid;
        const int p = row_position(a, n, rb, j);
        float nl = -INFINITY;
        if (h2o && fa.single) {
          // the caller's natural-log LSE of the query row (head g, position p)
          if (p >= 0) {
            const int g = j / a.P;
            const int64_t hq = static_cast<int64_t>(un.h) * a.G + g;
            const int64_t Hq = static_cast<int64_t>(a.Hkv) * a.G;
            const int64_t o = a.varlen ? (un.l * Hq + hq) * a.T + un.tok0 + p
                                       : ((static_cast<int64_t>(un.l) * a.b + un.s) * Hq + hq) * a.n_max + p;
            if (in_bounds(o, 1, fa.ext_h2o_lse, a.status)) nl = -__ldg(fa.h2o_lse + o) * kLog2e;
          }
        } else if (h2o) {
          const float2 ml = sh.merge[j];
          if (p >= 0 && ml.y > 0.f) nl = -(ml.x + log2f(ml.y));
        } else if (fa.single) {
          const int64_t o = static_cast<int64_t>(u) * kRowsMax + j;
          nl = (p >= 0 && in_bounds(o, 1, a.ext_lse2, a.status)) ? a.lse2[o] : -INFINITY;
        } else if (p >= 0) {
          // one online merge over the chunks, eight independent loads in flight
          const float2* part_j = a.partials + static_cast<int64_t>(u) * a.n_chunks * kRowsMax + j;
          float m = -INFINITY, s = 0.f;
          for (int c0 = 0; c0 < a.n_chunks; c0 += 8) {
            float2 v[8];
#pragma unroll
            for (int i = 0; i < 8; ++i)
              v[i] = (c0 + i < a.n_chunks &&
                      in_bounds(static_cast<int64_t>(u) * a.n_chunks * kRowsMax + j + (c0 + i) * kRowsMax, 1,
                                a.ext_partials, a.status))
                         ? __ldcg(&part_j[(c0 + i) * kRowsMax])
                         : make_float2(-INFINITY, 0.f);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              if (v[i].y > 0.f) {
                const float mn = fmaxf(m, v[i].x);
                s = s * exp2f(m - mn) + v[i].y * exp2f(v[i].x - mn);
                m = mn;
              }
            }
          }
          if (s > 0.f) nl = -(m + log2f(s));
        }
        sh.pos[j] = p;
        // -lse2_j / c1 as the sum of three bf16 parts (exact to ~2^-24); a row
        // without keys gets -1e30, whose exponential is 0
        const float x = nl > -INFINITY ? nl / c1 : -1.0e30f;
        const uint16_t h0 = bf16_bits_rn(x);
        const float r1 = x - bf16_value(h0);
        const uint16_t h1 = bf16_bits_rn(r1);
        const uint16_t h2 = bf16_bits_rn(r1 - bf16_value(h1));
        uint16_t* nlr = reinterpret_cast<uint16_t*>(sh.nlb);
        nlr[nl_elem(j, 0)] = h0;
        nlr[nl_elem(j, 1)] = h1;
        nlr[nl_elem(j, 2)] = h2;
        fence_proxy_async_smem();
      }
      mbar_arrive(sh.lse_ready);
      ok = __all_sync(0xffffffffu, mbar_wait(sh.lse_ready, ipop & 1, sh.abort_flag, a.status));
      if (!ok) break;

      // ---- pass 2: column sums of this thread's key over its rows
      int min_pos;
      bool all_rows;
      row_block_span(a, n, rb, &min_pos, &all_rows);
      const int64_t sbase = score_base(a, un, u);
      for (int kt = kt0; kt < kt1; ++kt, ++pair) {
        const int t = kt * kTileKeys + kl;
        const bool fast = all_rows && (kt * kTileKeys + kTileKeys - 1 <= min_pos);
        const int ab = pair & 1;
        if (ab != grp) continue;                   // the other group's tile
        ok = __all_sync(0xffffffffu, mbar_wait(&sh.acc_full[ab], (pair >> 1) & 1, sh.abort_flag, a.status));
        if (!ok) break;
        tc_fence_after();
        float colsum = 0.f;
        // drain the owned columns NC at a time (64 when they divide: two
        // loads in flight per wait, and the buffer released halfway)
        auto drain = [&](auto nc_tag) {
          constexpr int NC = decltype(nc_tag)::value;
          uint32_t r[NC];
          for (int h = 0; h < p2cols / NC; ++h) {
            tmem_load_cols<NC>(tmem + lane_base + ab * 256 + j0 + h * NC, r);
            if (h + 1 == p2cols / NC) {
              tc_fence_before();
              mbar_arrive(&sh.acc_empty[ab]);
            }
            // the accumulator holds S_jt - lse2_j / c1: the normaliser came in
            // through the extra k-step, so no per-row value is loaded here
            if (fast) {
              float2 acc[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f),
                               make_float2(0.f, 0.f)};
#pragma unroll
              for (int i = 0; i < NC; i += 8) {
#pragma unroll
                for (int k = 0; k < 4; ++k)
                  acc[k] = __fadd2_rn(acc[k], exp2x2(__fmul2_rn(bits2(r, i + 2 * k), cc)));
              }
              const float2 s2 = __fadd2_rn(__fadd2_rn(acc[0], acc[1]), __fadd2_rn(acc[2], acc[3]));
              colsum += s2.x + s2.y;
            } else {
              const int32_t* pp = sh.pos + j0 + h * NC;
              float s = 0.f;
#pragma unroll
              for (int i = 0; i < NC; ++i) {
                const float e = fast_exp2(__uint_as_float(r[i]) * c1);
                s += (t <= pp[i]) ? e : 0.f;
              }
              colsum += s;
            }
          }
        };
        if (p2cols % 64 == 0)
          drain(std::integral_constant<int, 64>{});
        else
          drain(std::integral_constant<int, 32>{});
        // add the group's two row halves of this key and write s(t)
        if (gp != 0) {
          ok = mbar_wait(&sh.red_empty[grp], (xchg & 1) ^ 1, sh.abort_flag, a.status);
          if (!ok) break;
          sh.red[grp * kTileKeys + kl] = colsum;
          mbar_arrive(&sh.red_full[grp]);
        } else {
          ok = mbar_wait(&sh.red_full[grp], xchg & 1, sh.abort_flag, a.status);
          if (!ok) break;
          const float total = colsum + sh.red[grp * kTileKeys + kl];
          mbar_arrive(&sh.red_empty[grp]);
          if (t < n && in_bounds(sbase + t, 1, a.ext_scores, a.status)) {
            if (h2o)
              atomicAdd(a.prepool + sbase + t, total);   // one query block's share
            else
              a.prepool[sbase + t] = total;
          }
        }
        ++xchg;
      }
      ++ipop;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// Log2-domain normaliser of every SnapKV window row: combined from the pass-1
// partials, or taken from a caller-supplied natural-log LSE.
__global__ void snapkv_lse_kernel(const ScoreArgs a, const float* __restrict__ lse_win) {
  const int64_t idx = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
  if (idx >= static_cast<int64_t>(a.n_units) * kRowsMax) return;
  const int u = static_cast<int>(idx / kRowsMax);
  const int j = static_cast<int>(idx % kRowsMax);
  const Unit un = decode_unit(a, u);
  const int p = row_position(a, un.n, 0, j);
  float out = INFINITY;
  if (p >= 0) {
    if (lse_win != nullptr) {
      const int g = j / a.P, i = j % a.P;
      const int64_t o =
          ((static_cast<int64_t>(un.l) * a.b + un.s) * (static_cast<int64_t>(a.Hkv) * a.G) +
           static_cast<int64_t>(un.h) * a.G + g) * a.W + i;
      if (in_bounds(o, 1, a.ext_lse_win, a.status)) out = lse_win[o] * kLog2e;
    } else {
      const int64_t p0 = static_cast<int64_t>(u) * a.n_chunks * kRowsMax + j;
      const float2* part = a.partials + p0;
      if (in_bounds(p0, static_cast<int64_t>(a.n_chunks - 1) * kRowsMax + 1, a.ext_partials, a.status)) {
        float m = -INFINITY;
        for (int c = 0; c < a.n_chunks; ++c) m = fmaxf(m, part[c * kRowsMax].x);
        if (m > -INFINITY) {
          float l = 0.f;
          for (int c = 0; c < a.n_chunks; ++c) {
            const float2 v = part[c * kRowsMax];
            if (v.y > 0.f) l += v.y * exp2f(v.x - m);
          }
          out = m + log2f(l);
        }
      }
    }
  }
  if (in_bounds(static_cast<int64_t>(u) * kRowsMax + j, 1, a.ext_lse2, a.status))
    a.lse2[static_cast<int64_t>(u) * kRowsMax + j] = -out;
}

// Stride-1 max-pool over each unit's score row, truncated at the sequence
// ends (Algorithm 1, pooling step).
__global__ void maxpool_kernel(const ScoreArgs a, const float* __restrict__ in,
                               float* __restrict__ out, int pool_k, int blocks_per_unit) {
  const int u = blockIdx.x / blocks_per_unit;
  const int part = blockIdx.x % blocks_per_unit;
  const Unit un = decode_unit(a, u);
  const int64_t base = score_base(a, un, u);
  const int h = pool_k / 2;
  for (int t = part * blockDim.x + threadIdx.x; t < un.n; t += blocks_per_unit * blockDim.x) {
    const int lo = max(0, t - h), hi = min(un.n - 1, t + h);
    if (!in_bounds(base + lo, hi - lo + 1, a.ext_scores, a.status)) continue;
    float m = in[base + lo];
    for (int x = lo + 1; x <= hi; ++x) m = fmaxf(m, in[base + x]);
    out[base + t] = m;
  }
}

}  // namespace

// ------------------------------------------------------------------ launch --

template <int D, int PASS>
static cudaError_t launch_pass(const CUtensorMap& kmap, const CUtensorMap& qmap,
                               const ScoreArgs& a, int grid, cudaStream_t stream) {
  using C = Cfg<D, PASS>;
  cudaError_t e = cudaFuncSetAttribute(attn_pass_kernel<D, PASS>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemAlloc);
  if (e != cudaSuccess) return e;
  attn_pass_kernel<D, PASS><<<grid, kThreads, C::kSmemAlloc, stream>>>(kmap, qmap, a);
  return cudaGetLastError();
}

cudaError_t launch_attn_pass(int pass, int d, const CUtensorMap& kmap, const CUtensorMap& qmap,
                             const ScoreArgs& a, int grid, cudaStream_t stream) {
  if (grid <= 0) return cudaSuccess;
  if (d == 128)
    return pass == 0 ? launch_pass<128, kPassRowstats>(kmap, qmap, a, grid, stream)
                     : launch_pass<128, kPassColsum>(kmap, qmap, a, grid, stream);
  return pass == 0 ? launch_pass<64, kPassRowstats>(kmap, qmap, a, grid, stream)
                   : launch_pass<64, kPassColsum>(kmap, qmap, a, grid, stream);
}

template <int D>
static cudaError_t launch_fused(const CUtensorMap& kmap, const CUtensorMap& qmap,
                                const FusedArgs& a, cudaStream_t stream) {
  using C = FCfg<D>;
  cudaError_t e = cudaFuncSetAttribute(snapkv_fused_kernel<D>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemAlloc);
  if (e != cudaSuccess) return e;
  int dev = 0, sms = 0, per_sm = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, snapkv_fused_kernel<D>, kThreads,
                                                         C::kSmemAlloc)) != cudaSuccess)
    return e;
  if (per_sm < 1) return cudaErrorInvalidConfiguration;
  // One CTA per SM, all resident at once (the per-unit arrival counters are
  // waited on), which the cooperative launch guarantees.  The grid is a
  // multiple of the chunks per unit so that items dealt round-robin put all
  // of a unit's chunks in the same round.
  const int nc = a.s.n_chunks;
  if (nc < 1 || nc > sms) return cudaErrorInvalidConfiguration;
  // (no more CTAs than items: a small batch does not set up idle CTAs; the
  // count stays a multiple of the chunks per unit)
  const int items = ((a.n_items + nc - 1) / nc) * nc;
  const int grid = std::min((sms / nc) * nc, std::max(items, nc));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(grid));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = C::kSmemAlloc;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  e = cudaLaunchKernelEx(&cfg, snapkv_fused_kernel<D>, kmap, qmap, a);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_snapkv_fused(int d, const CUtensorMap& kmap, const CUtensorMap& qmap,
                                const FusedArgs& a, cudaStream_t stream) {
  return d == 128 ? launch_fused<128>(kmap, qmap, a, stream) : launch_fused<64>(kmap, qmap, a, stream);
}

cudaError_t launch_snapkv_lse(const ScoreArgs& a, const float* lse_win, cudaStream_t stream) {
  const int64_t total = static_cast<int64_t>(a.n_units) * kRowsMax;
  if (total == 0) return cudaSuccess;
  const int threads = 256;
  const int blocks = static_cast<int>((total + threads - 1) / threads);
  snapkv_lse_kernel<<<blocks, threads, 0, stream>>>(a, lse_win);
  return cudaGetLastError();
}

cudaError_t launch_maxpool(const ScoreArgs& a, const float* in, float* out, int pool_k,
                           cudaStream_t stream) {
  if (a.n_units == 0 || a.n_max == 0) return cudaSuccess;
  const int per_unit = (a.n_max + 255) / 256;
  const int64_t grid = static_cast<int64_t>(per_unit) * a.n_units;
  maxpool_kernel<<<static_cast<unsigned>(grid), 256, 0, stream>>>(a, in, out, pool_k, per_unit);
  return cudaGetLastError();
}

}  // namespace rolekv
