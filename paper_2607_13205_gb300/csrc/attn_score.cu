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
//     thread-locally, so no cross-thread reduction is needed.
//
// In both passes one producer warp streams 128-key K tiles and 256-row query
// blocks into 128-byte-swizzled shared memory with TMA, one warp issues
// tcgen05.mma (bf16 operands, fp32 accumulators in tensor memory, two
// accumulator buffers) and eight epilogue warps drain the accumulators with
// tcgen05.ld.  Every wait is an mbarrier wait bounded in time.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "device_common.cuh"
#include "internal.h"

namespace rolekv {
namespace {

constexpr int kTileKeys = 128;
constexpr int kEpiWarps = 8;
constexpr int kProducerWarp = 8;
constexpr int kMmaWarp = 9;
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
  static constexpr int SQ = (PASS == kPassColsum) ? 2 : 1;
  static constexpr int SK = (PASS == kPassColsum) ? 2 : 4;
  static constexpr int kQOff = 0;
  static constexpr int kKOff = kQOff + SQ * kQSlotBytes;
  static constexpr int kLseOff = kKOff + SK * kKTileBytes;
  static constexpr int kPosOff = kLseOff + SQ * kRowsMax * 4;
  static constexpr int kRedOff = kPosOff + SQ * kRowsMax * 4;
  static constexpr int kMergeOff = kRedOff + kTileKeys * 4;
  static constexpr int kBarOff = kMergeOff + kRowsMax * 8;
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

__device__ __forceinline__ int num_row_blocks(const ScoreArgs& a, int n) {
  if (a.mode == kModeSnapKV) return n > 0 ? 1 : 0;
  return (n + a.P - 1) / a.P;
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
  } else if (pass == kPassRowstats) {
    const int rb = a.nrb_max - 1 - slot;        // longest query blocks first
    w.rb0 = rb;
    w.rb1 = (rb * a.P < n) ? rb + 1 : rb;
    const int kend = min(n, (rb + 1) * a.P);
    w.kt0 = 0;
    w.kt1 = (kend + kTileKeys - 1) / kTileKeys;
  } else {
    w.kt0 = slot;
    w.kt1 = (slot < ntiles) ? slot + 1 : slot;
    w.rb0 = (slot * kTileKeys) / a.P;
    w.rb1 = num_row_blocks(a, n);
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
  // Pass 2 of H2O streams query blocks against one key tile; every other
  // combination keeps one query block for the whole CTA.
  const bool q_streams = (PASS == kPassColsum) && (a.mode == kModeH2O);

  // ---- set-up: barriers, zeroed padding rows, tensor memory
  if (threadIdx.x == 0) {
    for (int i = 0; i < C::SK; ++i) {
      mbar_init(&sh.k_full[i], 1);
      mbar_init(&sh.k_empty[i], 1);
    }
    for (int i = 0; i < C::SQ; ++i) {
      mbar_init(&sh.q_full[i], 32);                     // every producer lane arrives
      mbar_init(&sh.q_empty[i], PASS == kPassColsum ? 1 + kEpiWarps * 32 : 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sh.acc_full[i], 1);
      mbar_init(&sh.acc_empty[i], kEpiWarps * 32);
    }
    mbar_init(sh.red_full, 128);
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
        if (PASS == kPassColsum) {
          const int64_t lrow =
              (static_cast<int64_t>(w.u) * (a.mode == kModeSnapKV ? 1 : a.nrb_max) + rb) * kRowsMax;
          for (int j = lane; j < kRowsMax; j += 32) {
            const int p = row_position(a, n, rb, j);
            sh.pos[slot * kRowsMax + j] = p;
            sh.lse[slot * kRowsMax + j] = (p >= 0) ? a.lse2[lrow + j] : INFINITY;
          }
        }
        if (lane == 0) {
          mbar_arrive_expect_tx(&sh.q_full[slot], static_cast<uint32_t>(a.nrows) * D * 2);
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
        } else {
          mbar_arrive(&sh.q_full[slot]);
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
    const int qd = warp & 3;
    const int hf = warp >> 2;
    const uint32_t lane_base = static_cast<uint32_t>(qd * 32) << 16;
    const float c1 = a.c1;
    int pair = 0;
    bool ok = true;
    if (PASS == kPassRowstats) {
      // The thread owns query row `row`.  With two row tiles each half of the
      // epilogue takes one tile; with one, the halves split the key columns
      // of every tile and merge at the end.
      const int row = (nrt == 2) ? hf * 128 + qd * 32 + lane : qd * 32 + lane;
      const int col0 = (nrt == 2) ? hf * 128 : hf * 64;
      const int key0 = (nrt == 2) ? 0 : hf * 64;
      const int nchunk = (nrt == 2) ? 4 : 2;
      const int rb = w.rb0;
      const int pos = (w.rb1 > w.rb0) ? row_position(a, n, rb, row) : -1;
      float m2 = -INFINITY, l = 0.f;
      for (int kt = w.kt0; kt < w.kt1 && ok; ++kt) {
        const int ab = pair & 1;
        ok = __all_sync(0xffffffffu, mbar_wait(&sh.acc_full[ab], (pair >> 1) & 1, sh.abort_flag, a.status));
        if (!ok) break;
        tc_fence_after();
        for (int c = 0; c < nchunk; ++c) {
          uint32_t r[32];
          __syncwarp();
          tmem_ld32(tmem + lane_base + ab * 256 + col0 + c * 32, r);
          tmem_wait_ld();
          tmem_reg_fence(r);
          const int t0 = kt * kTileKeys + key0 + c * 32;
          if (pos >= 0 && t0 <= pos) {
            const bool whole = (t0 + 31 <= pos);
            float mx = -INFINITY;
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if (whole || t0 + i <= pos) mx = fmaxf(mx, __uint_as_float(r[i]));
            const float mnew = fmaxf(m2, mx * c1);
            float acc = 0.f;
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const float e = fast_exp2(fmaf(__uint_as_float(r[i]), c1, -mnew));
              acc += (whole || t0 + i <= pos) ? e : 0.f;
            }
            l = l * fast_exp2(m2 - mnew) + acc;
            m2 = mnew;
          }
        }
        tc_fence_before();
        mbar_arrive(&sh.acc_empty[ab]);
        ++pair;
      }
      bool writer = (nrt == 2) || (hf == 0);
      if (nrt == 1 && ok) {
        // Merge the two column halves of each row.
        if (hf == 1) {
          sh.merge[row] = make_float2(m2, l);
          mbar_arrive(sh.red_full);
        } else {
          ok = mbar_wait(sh.red_full, 0, sh.abort_flag, a.status);
          if (ok) {
            const float2 o = sh.merge[row];
            const float mm = fmaxf(m2, o.x);
            if (mm > -INFINITY) {
              l = l * fast_exp2(m2 - mm) + o.y * fast_exp2(o.x - mm);
              m2 = mm;
            }
          }
        }
      }
      writer = writer && ok;
      if (writer) {
        if (a.mode == kModeSnapKV) {
          const int64_t slot = static_cast<int64_t>(w.u) * a.n_chunks + w.chunk;
          a.partials[slot * kRowsMax + row] = make_float2(m2, l);
          if (nrt == 1) a.partials[slot * kRowsMax + 128 + row] = make_float2(-INFINITY, 0.f);
        } else if (w.rb1 > w.rb0) {
          const int64_t o = (static_cast<int64_t>(w.u) * a.nrb_max + rb) * kRowsMax;
          a.lse2[o + row] = (l > 0.f) ? m2 + __log2f(l) : INFINITY;
          if (nrt == 1) a.lse2[o + 128 + row] = INFINITY;
        }
      }
    } else {
      // The thread owns key lane `kl` of the tile; the two halves split the
      // query rows and add up at the end of each key tile.
      const int kl = qd * 32 + lane;
      const int half_cols = a.nrows_pad / 2;
      const int nchunk = half_cols / 32;
      const int j0 = hf * half_cols;
      const int64_t sbase = score_base(a, w.unit, w.u);
      int quse = 0, xchg = 0;
      for (int kt = w.kt0; kt < w.kt1 && ok; ++kt) {
        const int t = kt * kTileKeys + kl;
        float colsum = 0.f;
        for (int rb = w.rb0; rb < w.rb1; ++rb) {
          const bool new_q = q_streams || kt == w.kt0;
          if (new_q) {
            // Acquire the producer's normalisers and positions for this block.
            ok = __all_sync(0xffffffffu, mbar_wait(&sh.q_full[quse % C::SQ], (quse / C::SQ) & 1,
                                                   sh.abort_flag, a.status));
            if (!ok) break;
            ++quse;
          }
          const int qslot = (quse - 1) % C::SQ;
          int min_pos;
          bool all_rows;
          row_block_span(a, n, rb, &min_pos, &all_rows);
          const bool fast = all_rows && (kt * kTileKeys + kTileKeys - 1 <= min_pos);
          const int ab = pair & 1;
          ok = __all_sync(0xffffffffu, mbar_wait(&sh.acc_full[ab], (pair >> 1) & 1, sh.abort_flag, a.status));
          if (!ok) break;
          tc_fence_after();
          const float* lse = sh.lse + qslot * kRowsMax + j0;
          const int32_t* pos = sh.pos + qslot * kRowsMax + j0;
          for (int c = 0; c < nchunk; ++c) {
            uint32_t r[32];
            __syncwarp();
            tmem_ld32(tmem + lane_base + ab * 256 + j0 + c * 32, r);
            tmem_wait_ld();
            tmem_reg_fence(r);
            float acc = 0.f;
            if (fast) {
#pragma unroll
              for (int i = 0; i < 32; i += 4) {
                const float4 L4 = *reinterpret_cast<const float4*>(lse + c * 32 + i);
                acc += fast_exp2(fmaf(__uint_as_float(r[i + 0]), c1, -L4.x));
                acc += fast_exp2(fmaf(__uint_as_float(r[i + 1]), c1, -L4.y));
                acc += fast_exp2(fmaf(__uint_as_float(r[i + 2]), c1, -L4.z));
                acc += fast_exp2(fmaf(__uint_as_float(r[i + 3]), c1, -L4.w));
              }
            } else {
#pragma unroll
              for (int i = 0; i < 32; ++i) {
                const float e = fast_exp2(fmaf(__uint_as_float(r[i]), c1, -lse[c * 32 + i]));
                acc += (t <= pos[c * 32 + i]) ? e : 0.f;
              }
            }
            colsum += acc;
          }
          tc_fence_before();
          mbar_arrive(&sh.acc_empty[ab]);
          if (q_streams || kt + 1 == w.kt1) mbar_arrive(&sh.q_empty[qslot]);
          ++pair;
        }
        if (!ok) break;
        // Add the two row halves of this key and write s(t).
        if (hf == 1) {
          ok = mbar_wait(sh.red_empty, (xchg & 1) ^ 1, sh.abort_flag, a.status);
          if (!ok) break;
          sh.red[kl] = colsum;
          mbar_arrive(sh.red_full);
        } else {
          ok = mbar_wait(sh.red_full, xchg & 1, sh.abort_flag, a.status);
          if (!ok) break;
          const float total = colsum + sh.red[kl];
          mbar_arrive(sh.red_empty);
          if (t < n) a.prepool[sbase + t] = total;
        }
        ++xchg;
      }
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
      out = lse_win[o] * kLog2e;
    } else {
      const float2* part = a.partials + static_cast<int64_t>(u) * a.n_chunks * kRowsMax + j;
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
  a.lse2[static_cast<int64_t>(u) * kRowsMax + j] = out;
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
