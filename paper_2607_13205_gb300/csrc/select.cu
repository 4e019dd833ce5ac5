// Role-conditional allocation and per-bucket top-k (Section 4.1, Algorithm 1):
// pool the scores (optional), count the roles, split the budget ceil(B n)
// across role buckets, and keep the top-q_r tokens of every bucket, ties to the
// lower index.  One CTA per (layer, sequence, KV head) holds the unit's keys
// in shared memory; everything after the fp32 -> ordered-key mapping is
// integer, so the kept set is bit-exact for a given score row.
//
// Slots.  Shared memory holds the unit in "slots": slot s is token s - off,
// where off = (start address of the score row / 4) mod 4, so that every group
// of four slots is one aligned 16-byte vector both in global and in shared
// memory.  Slots outside [off, off + n) have role 0xFF and are never kept.
//
// The threshold of each bucket is found by a radix descent over the keys'
// bits, most significant first:
//   pass 1  load, pool, key; per role, a histogram of the key's bits
//           30..31-NB (the top bit is shared by every key when all scores
//           have one sign): exponent and leading mantissa bits.  The role
//           counts are the histograms' sums.  Under GLOBAL there is one
//           bucket, so one histogram of every eligible token.
//   quotas  one warp, lane r for role r (water-filling, largest remainders).
//   first digit from the pass-1 histograms, per bucket; while the keys at
//           the threshold digits would overflow the list, a full pass over
//           the slots per 8 more bits.
//   pass 2  every token is decided (kept / dropped) unless its key prefix is
//           its bucket's threshold prefix; those "candidates" (a few
//           percent) go to a list in shared memory.
//   list    the remaining bits in 8-bit rounds over the list; ties at the
//           threshold are ranked in index order; the kept ones join the bits.
// A unit with a NaN, keys of both signs, or more candidates than the list
// holds 4 to 5 bits above the bottom takes the general path: four 8-bit
// rounds over all slots.
// Rows longer than kSmemMaxN tokens (streaming mode) do not keep their keys:
// every pass recomputes a group's pooled keys from the score row (read again
// from L2), the first-digit histograms count in 32 bits and a candidate-list
// entry carries its key beside (bucket << 24) | slot.
// Kept positions are then written in ascending order from a block-wide scan
// of the bit words.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "device_common.cuh"
#include "internal.h"

namespace rolekv {
namespace {

constexpr int kR = ROLEKV_MAX_ROLES;
constexpr uint32_t kCodeKeep = 0x40;   // the token's bucket keeps everything
constexpr uint32_t kCodeDrop = 0x80;   // no bucket keeps the token
// codes 0 .. kR-1: the token's bucket keeps only keys above a threshold
constexpr int kTieCap = 256;           // ranked ties held in shared memory

// Longest row whose keys a CTA holds in shared memory; longer rows take the
// streaming mode.
constexpr int kSmemMaxN = 40960;

// Groups (of four slots) reserved per CTA: n_max tokens plus up to three
// leading slots, rounded to a multiple of 32 groups so that the bit words
// (one per 8 groups) end on a 16-byte boundary.
__host__ __device__ inline int select_groups(int n_max) { return (((n_max + 3 + 3) / 4) + 31) & ~31; }
// Width of the first digit: 2^NB bins per role.
__host__ __device__ inline int first_digit_bits(int n_max) { return n_max > 16384 ? 11 : 10; }
// Bytes of the region that holds the pass-1 histograms (8 roles x 2^NB bins
// x 16-bit counts; 32-bit in streaming mode, where a bin can pass 65535),
// reused for the candidate list (4-byte entries; 8-byte in streaming mode).
__host__ __device__ inline size_t region_bytes(int n_max) {
  return static_cast<size_t>(kR) * (size_t{1} << first_digit_bits(n_max)) * (n_max > kSmemMaxN ? 4 : 2);
}

// Monotone map of a float to uint32 (larger float -> larger key); -0 is folded
// onto +0 so equal floats give equal keys.
__device__ __forceinline__ uint32_t ordered_key(float f) {
  if (f == 0.0f) f = 0.0f;
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float max3f(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// x << s, with every shift of 64 or more giving 0 (PTX clamps the amount).
__device__ __forceinline__ uint64_t shl64(uint64_t x, uint32_t s) {
  uint64_t r;
  asm("shl.b64 %0, %1, %2;" : "=l"(r) : "l"(x), "r"(s));
  return r;
}

__device__ __forceinline__ int warp_sum(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

struct SelShared {
  int64_t keep_off;
  int32_t count[kR];       // tokens per role
  int32_t quota[kR];       // q_b per bucket
  uint32_t prefix[kR];     // threshold key bits found so far
  int32_t need[kR];        // tokens equal to the prefix still to keep
  uint32_t thr[kR];        // keep iff key >= thr (ties ranked apart when partial)
  int32_t mode[kR];        // 0 none kept, 1 all kept, 2 threshold
  int32_t cand[kR];        // candidates after the first digit
  int32_t code_of_role[256];
  int32_t first_of_role[256];  // pass 2: keep iff first digit > it, candidate iff ==
  int32_t hist[kR][256];
  int32_t warp_tot[32];
  int32_t kept_role[kR];
  int32_t floor_role[kR];  // recency-floor tokens per role
  uint32_t ties[kTieCap];  // (bucket << 16) | slot of keys equal to a threshold
  uint32_t top_and, top_or;
  int32_t list_n, tie_n;
  int32_t nan_hint;        // a sum of the unit's scores was NaN
  int32_t nan_seen;        // a pooled window held a NaN
  int32_t any_threshold;
  int32_t general;         // take the full-pass descent
  uint32_t partial_ties;   // buckets with more threshold ties than slots left
  int32_t slack;           // SLACK policy: slots left to fill by score
  uint32_t elig_mask;      // roles taking part in the split (bit r)
  int32_t sfast;           // SLACK: the fill's first digit is known (below)
  uint32_t sprefix;        // SLACK: shared top bit and first digit of the fill threshold
  int32_t sneed;           // SLACK: tokens at that digit still to fill
};

// Slots 4g .. 4g+3 of a score row; slots outside [off, off + n) read -inf.
// sp + (4g - off) is 16-byte aligned by the choice of off.
__device__ __forceinline__ float4 load_slots(const float* sp, int off, int n, int g) {
  const int s0 = 4 * g - off;
  if (s0 >= 0 && s0 + 4 <= n) return __ldg(reinterpret_cast<const float4*>(sp + s0));
  float4 r;
  r.x = (s0 >= 0 && s0 < n) ? __ldg(sp + s0) : -INFINITY;
  r.y = (s0 + 1 >= 0 && s0 + 1 < n) ? __ldg(sp + s0 + 1) : -INFINITY;
  r.z = (s0 + 2 >= 0 && s0 + 2 < n) ? __ldg(sp + s0 + 2) : -INFINITY;
  r.w = (s0 + 3 >= 0 && s0 + 3 < n) ? __ldg(sp + s0 + 3) : -INFINITY;
  return r;
}

// Role bytes of slots 4g .. 4g+3 (0xFF outside the sequence).
__device__ __forceinline__ uint32_t load_roles(const uint8_t* rp, int off, int n, int g, bool vec) {
  const int s0 = 4 * g - off;
  if (vec && s0 >= 0 && s0 + 4 <= n) return __ldg(reinterpret_cast<const uint32_t*>(rp + s0));
  uint32_t w = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const int t = s0 + j;
    const uint32_t r = (t >= 0 && t < n) ? static_cast<uint32_t>(__ldg(rp + t)) : 0xFFu;
    w |= r << (8 * j);
  }
  return w;
}

struct UnitView {
  const float* sp;
  const uint8_t* rp;
  int off, n, ngroups;
  int nf;          // tokens before the recency floor (the floor is [nf, n))
  bool rvec;
};

// Bits j of the slots 4g+j (first token s0 = 4g - off) inside the recency
// floor [nf, n).
__device__ __forceinline__ uint32_t floor_bits(int s0, int nf, int n) {
  if (s0 + 4 <= nf || s0 >= n) return 0u;
  uint32_t m = 0;
#pragma unroll
  for (int j = 0; j < 4; ++j)
    if (s0 + j >= nf && s0 + j < n) m |= 1u << j;
  return m;
}

// Pass 1 for a pool half-width HW known at compile time.
template <int HW, int NT, bool GL, bool STREAM>
__device__ __forceinline__ void pass1(const UnitView& v, int n_roles, uint32_t ban, int nb,
                                      uint4* keys4, uint32_t* hist16, int32_t* floor_role,
                                      bool& nan_hint, uint32_t& top_and, uint32_t& top_or) {
  constexpr int NB = (HW + 3) / 4;   // neighbour groups on each side
  const int sh0 = 31 - nb;
  const uint32_t bmask = (1u << nb) - 1u;
  const int words_per_role = 1 << (nb - 1);
  for (int g = threadIdx.x; g < v.ngroups; g += NT) {
    // the role bytes are loaded with the scores, not after the pooling
    const uint32_t rw = load_roles(v.rp, v.off, v.n, g, v.rvec);
    float x[4 * (2 * NB + 1)];
#pragma unroll
    for (int o = -NB; o <= NB; ++o) {
      const float4 f = load_slots(v.sp, v.off, v.n, g + o);
      x[4 * (o + NB) + 0] = f.x;
      x[4 * (o + NB) + 1] = f.y;
      x[4 * (o + NB) + 2] = f.z;
      x[4 * (o + NB) + 3] = f.w;
    }
    const float* c = x + 4 * NB;
    const float sum = (c[0] + c[1]) + (c[2] + c[3]);
    nan_hint |= (sum != sum);
    uint32_t k[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      float m = c[j - HW];
#pragma unroll
      for (int o = -HW + 1; o <= HW; o += 2) {
        if (o < HW)
          m = max3f(m, c[j + o], c[j + o + 1]);
        else
          m = fmaxf(m, c[j + o]);
      }
      k[j] = ordered_key(m);
    }
    if (!STREAM) keys4[g] = make_uint4(k[0], k[1], k[2], k[3]);
    const uint32_t fb = floor_bits(4 * g - v.off, v.nf, v.n);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const uint32_t r = (rw >> (8 * j)) & 0xFFu;
      if ((fb >> j) & 1u) {                      // recency floor: kept, counted apart
        if (r < static_cast<uint32_t>(n_roles)) atomicAdd(&floor_role[r], 1);
      } else if (r < static_cast<uint32_t>(n_roles)) {
        top_and &= k[j];
        top_or |= k[j];
        const uint32_t bin = (k[j] >> sh0) & bmask;
        if (!GL || !((ban >> r) & 1u)) {
          if (STREAM)
            atomicAdd(&hist16[((GL ? 0u : r) << nb) + bin], 1u);   // 32-bit bins
          else
            atomicAdd(&hist16[(GL ? 0u : r) * words_per_role + (bin >> 1)], 1u << (16 * (bin & 1u)));
        }
      }
    }
  }
}

// Streaming mode: the four keys of group g recomputed from the score row, the
// same max-pool as pass 1 (stride 1, -inf outside the row, half-width hw);
// nan_aware: a window holding a NaN gives key 0 (below every other key).
__device__ __forceinline__ uint4 stream_group_keys(const UnitView& v, int g, int hw, bool nan_aware) {
  float x[20];
#pragma unroll
  for (int o = -2; o <= 2; ++o) {
    const float4 f = load_slots(v.sp, v.off, v.n, g + o);
    x[4 * (o + 2) + 0] = f.x;
    x[4 * (o + 2) + 1] = f.y;
    x[4 * (o + 2) + 2] = f.z;
    x[4 * (o + 2) + 3] = f.w;
  }
  uint32_t k[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    float m = x[8 + j];
    bool nanw = m != m;
#pragma unroll
    for (int d = 1; d <= 7; ++d) {
      if (d <= hw) {
        const float lo = x[8 + j - d], hi = x[8 + j + d];
        nanw |= (lo != lo) | (hi != hi);
        m = max3f(m, lo, hi);
      }
    }
    k[j] = (nan_aware && nanw) ? 0u : ordered_key(m);
  }
  return make_uint4(k[0], k[1], k[2], k[3]);
}

// Quotas of one sequence by warp 0, lane r for role r: water-filling of the
// weights over the role counts, then the integer remainders to the largest
// fractional parts (ties to the lower role), or under CEIL the ceiling of each
// share; the arithmetic stated in rolekv.h.
__device__ __forceinline__ int64_t sum8(int64_t v) {
  v += __shfl_xor_sync(0xffffffffu, v, 1);
  v += __shfl_xor_sync(0xffffffffu, v, 2);
  v += __shfl_xor_sync(0xffffffffu, v, 4);
  return v;
}

__device__ void quotas_warp(const SelectArgs& a, int lane, int64_t K_full, SelShared& S) {
  // every group of 8 lanes holds the 8 roles, so sums over a group are the
  // totals and all lanes take the same branches
  const int r = lane & (kR - 1);
  const bool valid = r < a.n_roles;
  const bool banned = valid && ((a.ban_mask >> r) & 1u);
  const int64_t cnt = valid ? S.count[r] : 0;
  // FAIR: every non-banned role weighted by its own token count
  const int64_t alpha = (a.policy == ROLEKV_POLICY_FAIR) ? ((valid && !banned) ? cnt : 0)
                                                         : a.alpha_fx[r];
  int64_t q = 0, bsize = 0;
  if (a.policy == ROLEKV_POLICY_GLOBAL) {
    const int64_t elig = S.count[0];   // every eligible token, counted in row 0
    if (r == 0) {
      q = K_full < elig ? K_full : elig;
      bsize = elig;
    }
  } else {
    bool live = valid && alpha > 0 && cnt > 0;
    const unsigned elig_bits = __ballot_sync(0xffffffffu, live) & 0xFFu;
    const int64_t elig = sum8(live ? cnt : 0);
    const int64_t k_all = K_full < elig ? K_full : elig;
    int64_t left = k_all;
    // SLACK: one round of the split, no water-filling (the slack of saturated
    // buckets is filled by score afterwards)
    for (int it = 0; it <= kR && a.policy != ROLEKV_POLICY_SLACK; ++it) {
      const int64_t A = sum8(live ? alpha : 0);
      if (A == 0) break;
      const bool sat = live && alpha * left >= cnt * A;
      if (!__any_sync(0xffffffffu, sat)) break;
      if (sat) {
        q = cnt;
        live = false;
      }
      left -= sum8(sat ? cnt : 0);
    }
    const int64_t A = sum8(live ? alpha : 0);
    if (a.policy == ROLEKV_POLICY_CEIL) {
      // Algorithm 1 read literally: each unsaturated bucket takes the ceiling
      // of its share (the total may exceed the budget; the rows are wider)
      if (live && A != 0) q = (alpha * left + A - 1) / A;
    } else {
      int64_t rem = -1;
      if (live && A != 0) {
        q = alpha * left / A;
        rem = alpha * left % A;
      }
      const int64_t extra = left - sum8(live ? q : 0);
      int rank = 0;
#pragma unroll
      for (int x = 0; x < kR; ++x) {
        const int64_t rx = __shfl_sync(0xffffffffu, rem, x);
        const int lx = __shfl_sync(0xffffffffu, static_cast<int>(live), x);
        if (lx && (rx > rem || (rx == rem && x < r))) ++rank;
      }
      if (live && A != 0 && rank < extra) q += 1;
    }
    if (a.policy == ROLEKV_POLICY_SLACK) {
      q = q < cnt ? q : cnt;
      const int64_t slack = k_all - sum8(q);
      if (lane == 0) {
        S.slack = static_cast<int32_t>(slack);
        S.elig_mask = elig_bits;
      }
    }
    bsize = cnt;
  }
  int mode = 0;
  if (lane < kR) {
    mode = (q <= 0) ? 0 : (q >= bsize ? 1 : 2);
    S.quota[r] = static_cast<int32_t>(q);
    S.mode[r] = mode;
    S.prefix[r] = 0;
    S.need[r] = static_cast<int32_t>(q);
    S.thr[r] = 0xFFFFFFFFu;   // above every key; set by the last radix round
    S.cand[r] = 0;
  }
  const bool any = __any_sync(0xffffffffu, mode == 2);
  if (lane == 0) {
    S.any_threshold = any;
    S.partial_ties = 0;
    S.list_n = 0;
    S.tie_n = 0;
  }
}

// The bucket's key among its remaining candidates with need[b] keys at or
// above it: warp b reads the histogram of the digit at `shift` (clearing it),
// finds the digit where the count from the top reaches need[b], appends it to
// prefix[b] and subtracts the keys above.  At shift 0 the prefix is the
// q_b-th largest key; thr[b] and the partial-tie flag are then set.
__device__ void descend(SelShared& S, int b, int lane, int shift) {
  int c[8];
  int mine = 0;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    c[i] = S.hist[b][lane * 8 + i];
    S.hist[b][lane * 8 + i] = 0;
    mine += c[i];
  }
  int incl = mine;   // tokens whose digit is in this lane's range or above
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int v = __shfl_down_sync(0xffffffffu, incl, o);
    if (lane + o < 32) incl += v;
  }
  const int above = incl - mine;
  const int need = S.need[b];
  int found = -1, gt_before = 0, at_digit = 0;
  if (above < need && above + mine >= need) {
    int acc = above;
#pragma unroll
    for (int i = 7; i >= 0; --i) {
      if (found < 0 && acc + c[i] >= need) {
        found = lane * 8 + i;
        gt_before = acc;
        at_digit = c[i];
      }
      acc += c[i];
    }
  }
  const unsigned who = __ballot_sync(0xffffffffu, found >= 0);
  const int src = who ? __ffs(who) - 1 : 0;
  const int fd = __shfl_sync(0xffffffffu, found, src);
  const int gb = __shfl_sync(0xffffffffu, gt_before, src);
  const int ad = __shfl_sync(0xffffffffu, at_digit, src);
  if (lane == 0 && who != 0) {
    const uint32_t prefix = S.prefix[b] | (static_cast<uint32_t>(fd) << shift);
    const int need2 = need - gb;
    S.prefix[b] = prefix;
    S.need[b] = need2;
    S.cand[b] = ad;
    if (shift == 0) {
      // ad keys of the bucket equal the threshold; need2 of them are kept
      S.thr[b] = (need2 >= ad) ? prefix : prefix + 1u;
      if (need2 < ad) atomicOr(&S.partial_ties, 1u << b);
    }
  }
}

// First digit (bits 30..31-nb, the shared top bit above them) of bucket b from
// the per-role 16-bit histograms of pass 1; the bucket's histogram is the sum
// over its roles.  Lane L owns a contiguous range of bins: the lanes' totals
// (read in a rotated order, so that the lanes hit different banks) locate the
// lane holding the threshold, then the warp splits that lane's words.
template <int NB>
__device__ void descend_first(const SelectArgs& a, SelShared& S, const uint32_t* hist16, int b,
                              int lane) {
  constexpr int nb = NB;
  constexpr int wpl = 1 << (nb - 6);   // histogram words (two bins each) per lane
  constexpr int wpr = 1 << (nb - 1);   // words per role
  // counts of bins 2w (low half) and 2w+1 (high half); a bin holds at most
  // n < 65536 tokens, so the halves never carry
  const uint32_t* h0 = hist16 + b * wpr;
  int mine = 0;
#pragma unroll
  for (int i = 0; i < wpl; ++i) {
    const uint32_t x = h0[lane * wpl + ((i + lane) & (wpl - 1))];
    mine += static_cast<int>((x & 0xFFFFu) + (x >> 16));
  }
  int incl = mine;   // tokens in this lane's bins or above
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int v = __shfl_down_sync(0xffffffffu, incl, o);
    if (lane + o < 32) incl += v;
  }
  const int above = incl - mine;
  const int need = S.need[b];
  const unsigned who = __ballot_sync(0xffffffffu, above < need && above + mine >= need);
  if (who == 0) {
    if (lane == 0) S.general = 1;   // counts disagree with the quota: let the full path decide
    return;
  }
  const int F = __ffs(who) - 1;
  const int aboveF = __shfl_sync(0xffffffffu, above, F);
  const int needF = need - aboveF;
  const uint32_t x = lane < wpl ? h0[F * wpl + lane] : 0u;
  const int lo = static_cast<int>(x & 0xFFFFu), hi = static_cast<int>(x >> 16);
  const int pair = lo + hi;
  int incl2 = pair;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int v = __shfl_down_sync(0xffffffffu, incl2, o);
    if (lane + o < 32) incl2 += v;
  }
  const int above2 = incl2 - pair;
  const unsigned who2 = __ballot_sync(0xffffffffu, above2 < needF && above2 + pair >= needF);
  if (who2 == 0) {
    if (lane == 0) S.general = 1;
    return;
  }
  if (lane == __ffs(who2) - 1) {
    const int w = F * wpl + lane;
    int fd, gb, ad;
    if (above2 + hi >= needF) {
      fd = 2 * w + 1;
      gb = aboveF + above2;
      ad = hi;
    } else {
      fd = 2 * w;
      gb = aboveF + above2 + hi;
      ad = lo;
    }
    const int sh0 = 31 - nb;
    S.prefix[b] = (S.top_and & 0x80000000u) | (static_cast<uint32_t>(fd) << sh0);
    S.need[b] = need - gb;
    S.cand[b] = ad;
  }
}

// SLACK policy: the first digit of the fill threshold, from the same pass-1
// histograms, once every bucket's first digit is known.  The tokens the fill
// ranks are the eligible ones no bucket keeps; per first-digit bin they are
// a role's whole bin (its bucket keeps nothing, or the bin lies below the
// bucket's digit), none (the bucket keeps the bin), or the bin less the
// need[b] tokens the bucket keeps at its own digit.  Every thread counts a
// few bins into `cnt` (shared memory, 2^NB ints); then warp 0 locates the
// bin holding the slack-th token from the top: each lane sums a contiguous
// range, the lanes' totals from the top locate the range, and the warp
// splits that range.  On success sprefix / sneed are set and sfast = 1;
// otherwise the fill takes its full-pass rounds.  Every thread calls it.
template <int NB, int NT>
__device__ void slack_first(const SelectArgs& a, SelShared& S, const uint32_t* hist16, int* cnt,
                            int list_cap) {
  constexpr int nbins = 1 << NB;
  constexpr int bpl = nbins / 32;        // bins per lane
  constexpr int wpr = 1 << (NB - 1);     // histogram words (two bins each) per role
  constexpr int sh0 = 31 - NB;
  const int tid = threadIdx.x, lane = tid & 31;
  for (int x = tid; x < nbins; x += NT) {
    int c = 0;
    for (int r = 0; r < a.n_roles; ++r) {
      if (!((S.elig_mask >> r) & 1u)) continue;
      const uint32_t code = static_cast<uint32_t>(S.code_of_role[r]);
      if (code == kCodeKeep) continue;
      const uint32_t w = hist16[r * wpr + (x >> 1)];
      const int h = static_cast<int>((x & 1) ? (w >> 16) : (w & 0xFFFFu));
      if (code >= static_cast<uint32_t>(kR)) {
        c += h;                                  // its bucket keeps nothing
      } else {
        const int D = static_cast<int>((S.prefix[code] >> sh0) & (nbins - 1));
        c += x < D ? h : (x == D ? h - S.need[code] : 0);
      }
    }
    cnt[x] = c;
  }
  __syncthreads();
  if (tid < 32) {
    const int need = S.slack;
    int mine = 0;
#pragma unroll 8
    for (int i = 0; i < bpl; ++i) mine += cnt[lane * bpl + ((i + lane) & (bpl - 1))];
    int incl = mine;                             // tokens in this lane's bins or above
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_down_sync(0xffffffffu, incl, o);
      if (lane + o < 32) incl += v;
    }
    const int above = incl - mine;
    const unsigned who = __ballot_sync(0xffffffffu, above < need && above + mine >= need);
    if (who != 0) {
      const int F = __ffs(who) - 1;
      const int aboveF = __shfl_sync(0xffffffffu, above, F);
      const int needF = need - aboveF;
      // the winning range split over the warp: bpl / 32 bins a lane
      constexpr int per = bpl / 32 > 0 ? bpl / 32 : 1;
      int c2[per];
      int part = 0;
#pragma unroll
      for (int i = 0; i < per; ++i) {
        c2[i] = (lane * per + i < bpl) ? cnt[F * bpl + lane * per + i] : 0;
        part += c2[i];
      }
      int incl2 = part;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int v = __shfl_down_sync(0xffffffffu, incl2, o);
        if (lane + o < 32) incl2 += v;
      }
      const int above2 = incl2 - part;
      const unsigned who2 = __ballot_sync(0xffffffffu, above2 < needF && above2 + part >= needF);
      if (who2 != 0 && lane == __ffs(who2) - 1) {
        int acc = above2, fd = -1, nd = 0, at = 0;
#pragma unroll
        for (int i = per - 1; i >= 0; --i) {
          if (fd < 0 && acc + c2[i] >= needF) {
            fd = F * bpl + lane * per + i;
            nd = needF - acc;
            at = c2[i];
          }
          acc += c2[i];
        }
        if (fd >= 0 && at <= list_cap) {
          S.sprefix = (S.top_and & 0x80000000u) | (static_cast<uint32_t>(fd) << sh0);
          S.sneed = nd;
          S.sfast = 1;
        }
      }
    }
  }
  __syncthreads();
  for (int x = tid; x < nbins; x += NT) cnt[x] = 0;
  __syncthreads();
}

// descend_first for the streaming mode's 32-bit bins: lane L owns bins
// L * 2^NB / 32 ..; the lanes' totals locate the lane holding the threshold,
// then the warp splits that lane's bins (at most 64, two per lane).
template <int NB>
__device__ void descend_first32(const SelectArgs& a, SelShared& S, const uint32_t* hist32, int b,
                                int lane) {
  constexpr int bpl = 1 << (NB - 5);   // bins per lane
  const uint32_t* h0 = hist32 + (b << NB);
  int mine = 0;
#pragma unroll 8
  for (int i = 0; i < bpl; ++i) mine += static_cast<int>(h0[lane * bpl + ((i + lane) & (bpl - 1))]);
  int incl = mine;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int v = __shfl_down_sync(0xffffffffu, incl, o);
    if (lane + o < 32) incl += v;
  }
  const int above = incl - mine;
  const int need = S.need[b];
  const unsigned who = __ballot_sync(0xffffffffu, above < need && above + mine >= need);
  if (who == 0) {
    if (lane == 0) S.general = 1;
    return;
  }
  const int F = __ffs(who) - 1;
  const int aboveF = __shfl_sync(0xffffffffu, above, F);
  const int needF = need - aboveF;
  // lane L takes bins F * bpl + 2L, 2L + 1 (descending order: the higher bin first)
  const int i0 = 2 * lane;
  const int lo = i0 < bpl ? static_cast<int>(h0[F * bpl + i0]) : 0;
  const int hi = i0 + 1 < bpl ? static_cast<int>(h0[F * bpl + i0 + 1]) : 0;
  const int pair = lo + hi;
  int incl2 = pair;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int v = __shfl_down_sync(0xffffffffu, incl2, o);
    if (lane + o < 32) incl2 += v;
  }
  const int above2 = incl2 - pair;
  const unsigned who2 = __ballot_sync(0xffffffffu, above2 < needF && above2 + pair >= needF);
  if (who2 == 0) {
    if (lane == 0) S.general = 1;
    return;
  }
  if (lane == __ffs(who2) - 1) {
    const int bin0 = F * bpl + i0;
    int fd, gb, ad;
    if (above2 + hi >= needF) {
      fd = bin0 + 1;
      gb = aboveF + above2;
      ad = hi;
    } else {
      fd = bin0;
      gb = aboveF + above2 + hi;
      ad = lo;
    }
    const int sh0 = 31 - NB;
    S.prefix[b] = (S.top_and & 0x80000000u) | (static_cast<uint32_t>(fd) << sh0);
    S.need[b] = need - gb;
    S.cand[b] = ad;
  }
}

// Exclusive prefix, in slot order, of popc(mask_of(q)) over the bit words
// q < nwords: warp w walks a contiguous range of words (a multiple of 32), the
// warps' totals are combined through shared memory, and body(q, mask, rank of
// the word's first set bit) runs once per word.  Returns the total.  Every
// thread of the CTA must call it.
template <int NT, class MaskF, class BodyF>
__device__ int scan_words(int nwords, MaskF mask_of, BodyF body, int32_t* warp_tot) {
  constexpr int NW = NT / 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int wseg = ((nwords + NW - 1) / NW + 31) & ~31;
  const int q_begin = warp * wseg;
  const int q_end = min(nwords, q_begin + wseg);
  int tot = 0;
  for (int q0 = q_begin; q0 < q_end; q0 += 32) {
    const int q = q0 + lane;
    if (q < q_end) tot += __popc(mask_of(q));
  }
  tot = warp_sum(tot);
  if (lane == 0) warp_tot[warp] = tot;
  __syncthreads();
  int base = warp_sum(lane < warp ? warp_tot[lane] : 0);
  const int total = warp_sum(lane < NW ? warp_tot[lane] : 0);
  for (int q0 = q_begin; q0 < q_end; q0 += 32) {
    const int q = q0 + lane;
    const uint32_t m = q < q_end ? mask_of(q) : 0u;
    const int c = __popc(m);
    int incl = c;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int v = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += v;
    }
    if (q < q_end) body(q, m, base + incl - c);
    base += __shfl_sync(0xffffffffu, incl, 31);
  }
  __syncthreads();
  return total;
}

// Keep bits of slots 4g .. 4g+3 (bit j = slot 4g+j) packed into one 32-bit
// word per 8 lanes; the lane with (lane & 7) == 0 stores word g / 8.
__device__ __forceinline__ void store_bits(uint32_t* bits, int g, int nwords, int lane, uint32_t m4) {
  uint32_t x = m4 << (4 * (lane & 7));
  x |= __shfl_xor_sync(0xffffffffu, x, 1);
  x |= __shfl_xor_sync(0xffffffffu, x, 2);
  x |= __shfl_xor_sync(0xffffffffu, x, 4);
  if ((lane & 7) == 0 && g < 8 * nwords) bits[g >> 3] = x;
}

template <int NT, bool STREAM>
__global__ void __launch_bounds__(NT, 1024 / NT) select_kernel(const SelectArgs a) {
  constexpr int NW = NT / 32;
  extern __shared__ __align__(16) uint8_t dyn[];
  __shared__ SelShared S;
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const int u = blockIdx.x;
  const int h = u % a.Hkv;
  const int s = (u / a.Hkv) % a.b;
  const int l = u / (a.Hkv * a.b);
  int n;
  int64_t tok0;
  if (a.varlen) {
    tok0 = a.cu_seqlens[s];
    n = a.cu_seqlens[s + 1] - a.cu_seqlens[s];
  } else {
    tok0 = 0;
    n = a.n_max;
  }
  const int64_t sbase =
      a.varlen ? (static_cast<int64_t>(l) * a.Hkv + h) * a.T + tok0 : static_cast<int64_t>(u) * a.n_max;
  const int64_t rbase = a.varlen ? tok0 : static_cast<int64_t>(s) * a.n_max;
  const int64_t K_s = kept_slots(n, a.budget_fx);              // the budget
  const int64_t width = kept_rows(n, a.budget_fx, a.kept_extra); // the kept row

  UnitView v;
  v.sp = a.scores + sbase;
  v.rp = a.roles + rbase;
  v.off = static_cast<int>((reinterpret_cast<uintptr_t>(v.sp) >> 2) & 3);
  v.n = n;
  const int nslots = v.off + n;
  v.ngroups = (nslots + 3) >> 2;
  v.rvec = ((reinterpret_cast<uintptr_t>(v.rp) - static_cast<uintptr_t>(v.off)) & 3u) == 0;
  const int64_t n_floor = a.keep_last < n ? (a.keep_last < K_s ? a.keep_last : K_s)
                                          : (n < K_s ? n : K_s);
  v.nf = n - static_cast<int>(n_floor);
  const int off = v.off, ngroups = v.ngroups;
  const int nwords = (nslots + 31) >> 5;
  const int iters = (ngroups + NT - 1) / NT;
  const int nb = first_digit_bits(a.n_max);
  const int groups_alloc = select_groups(a.n_max);
  // keys (in-memory mode only), keep bits, then the histogram / list region
  uint4* keys4 = reinterpret_cast<uint4*>(dyn);
  const uint32_t* keys = reinterpret_cast<const uint32_t*>(keys4);
  uint32_t* bits = reinterpret_cast<uint32_t*>(dyn + (STREAM ? 0 : static_cast<size_t>(groups_alloc) * 16));
  uint32_t* region = bits + groups_alloc / 8;   // 16-byte aligned (groups_alloc % 32 == 0)
  uint32_t* hist16 = region;                    // pass 1 histograms
  uint32_t* list = region;                      // then the candidate list
  const int list_cap = static_cast<int>(region_bytes(a.n_max) / (STREAM ? 8 : 4));
  const bool global = a.policy == ROLEKV_POLICY_GLOBAL;
  const int hw = a.pool_k / 2;
  // a group's four keys: held (in-memory mode) or recomputed from the scores
  bool nan_keys = false;                        // streaming mode: NaN windows give key 0
  auto kv_of = [&](int g) -> uint4 {
    if constexpr (STREAM) return stream_group_keys(v, g, hw, nan_keys);
    else return keys4[g];
  };

  if (tid < kR) {
    S.count[tid] = 0;
    S.kept_role[tid] = 0;
    S.floor_role[tid] = 0;
  }
  if (tid == 0) {
    S.nan_hint = 0;
    S.nan_seen = 0;
    S.general = 0;
    S.top_and = 0xFFFFFFFFu;
    S.top_or = 0u;
    S.slack = 0;
    S.elig_mask = 0u;
    S.sfast = 0;
  }
  for (int x = tid; x < kR * 256; x += NT) (&S.hist[0][0])[x] = 0;
  {
    uint4* r4 = reinterpret_cast<uint4*>(region);
    const int n4 = static_cast<int>(region_bytes(a.n_max) / 16);
    for (int x = tid; x < n4; x += NT) r4[x] = make_uint4(0u, 0u, 0u, 0u);
  }

  // ---- offset of this unit's kept row
  {
    int64_t part = 0;
    if (a.varlen) {
      for (int x = tid; x < s; x += NT)
        part += kept_rows(a.cu_seqlens[x + 1] - a.cu_seqlens[x], a.budget_fx, a.kept_extra);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
    __shared__ int64_t red64[NW];
    if (lane == 0) red64[warp] = part;
    __syncthreads();
    if (tid == 0) {
      int64_t cu = 0;
      for (int w = 0; w < NW; ++w) cu += red64[w];
      S.keep_off = a.varlen ? (static_cast<int64_t>(l) * a.Hkv + h) * a.Ktot + cu
                            : static_cast<int64_t>(u) * a.K_dense;
    }
  }

  // Checked build: the unit's score row (and mask row), role row, kept row
  // and per-role counts lie inside the extents the call's shapes give, or the
  // whole unit is skipped.
#ifdef ROLEKV_CHECKED
  __syncthreads();
  if (!(in_bounds(sbase, n, a.ext_scores, nullptr) && in_bounds(rbase, n, a.ext_roles, nullptr) &&
        in_bounds(S.keep_off, width, a.ext_keep, nullptr) &&
        (a.kept_per_role == nullptr ||
         in_bounds(static_cast<int64_t>(u) * a.n_roles, a.n_roles, static_cast<int64_t>(a.n_units) * a.n_roles,
                   nullptr)))) {
    if (tid == 0 && a.status != nullptr) atomicOr(a.status, ROLEKV_STATUS_BOUNDS);
    return;
  }
#endif

  // ---- pass 1: load, pool, key, first-digit histograms
  {
    bool nan_hint = false;
    uint32_t tand = 0xFFFFFFFFu, tor = 0u;
    // GLOBAL: one histogram (row 0) of every eligible token; otherwise one
    // row per role
#define ROLEKV_PASS1(HWV)                                                                           \
  (global ? pass1<HWV, NT, true, STREAM>(v, a.n_roles, a.ban_mask, nb, keys4, hist16, S.floor_role, \
                                         nan_hint, tand, tor)                                       \
          : pass1<HWV, NT, false, STREAM>(v, a.n_roles, a.ban_mask, nb, keys4, hist16, S.floor_role, \
                                          nan_hint, tand, tor))
    switch (a.pool_k >> 1) {
      case 0: ROLEKV_PASS1(0); break;
      case 1: ROLEKV_PASS1(1); break;
      case 2: ROLEKV_PASS1(2); break;
      case 3: ROLEKV_PASS1(3); break;
      case 4: ROLEKV_PASS1(4); break;
      case 5: ROLEKV_PASS1(5); break;
      case 6: ROLEKV_PASS1(6); break;
      default: ROLEKV_PASS1(7); break;
    }
#undef ROLEKV_PASS1
    tand = __reduce_and_sync(0xffffffffu, tand);
    tor = __reduce_or_sync(0xffffffffu, tor);
    const bool nh = __any_sync(0xffffffffu, nan_hint);
    if (lane == 0) {
      atomicAnd(&S.top_and, tand);
      atomicOr(&S.top_or, tor);
      if (nh) S.nan_hint = 1;
    }
  }
  __syncthreads();

  // Role counts: the sums of the roles' histograms (a warp's 32 words belong
  // to one role); GLOBAL: the eligible total, in count[0].
  {
    const int wpr = STREAM ? (1 << nb) : (1 << (nb - 1));   // words per role
    const int lwpr = STREAM ? nb : nb - 1;
    for (int x0 = warp * 32; x0 < (global ? 1 : a.n_roles) * wpr; x0 += NT) {
      const uint32_t w = hist16[x0 + lane];
      const int c = warp_sum(STREAM ? static_cast<int>(w) : static_cast<int>((w & 0xFFFFu) + (w >> 16)));
      if (lane == 0 && c) atomicAdd(&S.count[x0 >> lwpr], c);
    }
  }

  // A NaN score (or +inf and -inf in one group): redo the keys one token at a
  // time, a window holding a NaN giving the lowest key (streaming mode: every
  // later recomputation of the keys does so).
  if (STREAM) nan_keys = S.nan_hint != 0;
  if (STREAM && S.nan_hint) {
    bool seen = false;
    for (int t = tid; t < n; t += NT) seen |= isnan(__ldg(v.sp + t));
    if (__any_sync(0xffffffffu, seen) && lane == 0) S.nan_seen = 1;
  }
  if (!STREAM && S.nan_hint) {
    const int hw = a.pool_k / 2;
    uint32_t* kw = reinterpret_cast<uint32_t*>(keys4);
    bool seen = false;
    for (int t = tid; t < n; t += NT) {
      const int lo = max(0, t - hw), hi = min(n - 1, t + hw);
      float m = __ldg(v.sp + lo);
      bool nan_w = isnan(m);
      for (int x = lo + 1; x <= hi; ++x) {
        const float f = __ldg(v.sp + x);
        nan_w |= isnan(f);
        m = fmaxf(m, f);
      }
      seen |= nan_w;
      kw[t + off] = nan_w ? 0u : ordered_key(m);
    }
    if (__any_sync(0xffffffffu, seen) && lane == 0) S.nan_seen = 1;
  }
  __syncthreads();

  // ---- quotas and the role -> code table
  if (warp == 0) quotas_warp(a, lane, K_s - n_floor, S);
  __syncthreads();
  for (int x = tid; x < 256; x += NT) {
    uint32_t code = kCodeDrop;
    if (x < a.n_roles && !((a.ban_mask >> x) & 1u)) {
      const int b = (a.policy == ROLEKV_POLICY_GLOBAL) ? 0 : x;
      code = S.mode[b] == 2 ? static_cast<uint32_t>(b) : (S.mode[b] == 1 ? kCodeKeep : kCodeDrop);
    }
    S.code_of_role[x] = static_cast<int32_t>(code);
  }
  const bool any_thr = S.any_threshold != 0;
  if (tid == 0 && (S.nan_hint || ((S.top_and ^ S.top_or) & 0x80000000u))) S.general = 1;
  __syncthreads();

  // ---- first digit per bucket
  if (any_thr && !S.general) {
    if (warp < kR && S.mode[warp] == 2) {
      if (STREAM)
        descend_first32<11>(a, S, hist16, warp, lane);
      else if (nb == 11)
        descend_first<11>(a, S, hist16, warp, lane);
      else
        descend_first<10>(a, S, hist16, warp, lane);
    }
    __syncthreads();
  }
  // SLACK: the fill's first digit from the same histograms, before their
  // region becomes the candidate list (in-memory rows; 16-bit bins)
  if (!STREAM && S.slack > 0 && !S.general) {
    // (S.hist, zero until the refinement rounds, serves as the bin counts)
    static_assert(kR * 256 >= 2048, "bin counts for an 11-bit digit");
    if (nb == 11)
      slack_first<11, NT>(a, S, hist16, &S.hist[0][0], list_cap);
    else
      slack_first<10, NT>(a, S, hist16, &S.hist[0][0], list_cap);
  }
  // While the keys at the buckets' first digits overflow the list (scores in
  // a narrow range, such as page bounds), one full pass per 8 more bits.
  int shd = 31 - nb;   // key bits below the decided prefixes
  if (any_thr && !S.general) {
    auto cand_total = [&]() {
      int t = 0;
      for (int b = 0; b < kR; ++b) t += S.mode[b] == 2 ? S.cand[b] : 0;
      return t;
    };
    while (cand_total() > list_cap && shd > 8) {
      const int shift = shd - 8;
      for (int i = 0; i < iters; ++i) {
        const int g = i * NT + tid;
        if (g >= ngroups) break;
        const uint4 kv = kv_of(g);
        const uint32_t kk[4] = {kv.x, kv.y, kv.z, kv.w};
        const uint32_t rw = load_roles(v.rp, off, n, g, v.rvec);
        const uint32_t fb = floor_bits(4 * g - off, v.nf, n);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t c = static_cast<uint32_t>(S.code_of_role[(rw >> (8 * j)) & 0xFFu]);
          if (c >= static_cast<uint32_t>(kR) || ((fb >> j) & 1u)) continue;
          if ((kk[j] >> shd) != (S.prefix[c] >> shd)) continue;
          atomicAdd(&S.hist[c][(kk[j] >> shift) & 0xFFu], 1);
        }
      }
      __syncthreads();
      if (warp < kR && S.mode[warp] == 2) descend(S, warp, lane, shift);
      __syncthreads();
      shd = shift;
    }
    if (tid == 0 && cand_total() > list_cap) S.general = 1;
    __syncthreads();
  }

  if (!S.general) {
    for (int x = tid; x < 256; x += NT) {
      const uint32_t code = static_cast<uint32_t>(S.code_of_role[x]);
      S.first_of_role[x] = code == kCodeKeep                  ? -1
                           : code < static_cast<uint32_t>(kR) ? static_cast<int32_t>(S.prefix[code] >> shd)
                                                               : 0x7FFFFFFF;
    }
    __syncthreads();
    // ---- pass 2: decide every token outside its bucket's threshold digit,
    // list the rest
    // roles are read two iterations ahead of their use (they come from L2)
    auto roles_of = [&](int i) {
      const int g = i * NT + tid;
      return (i < iters && g < ngroups) ? load_roles(v.rp, off, n, g, v.rvec) : 0xFFFFFFFFu;
    };
    uint32_t r_next = roles_of(0), r_after = roles_of(1);
    for (int i = 0; i < iters; ++i) {
      const int g = i * NT + tid;
      const uint32_t rw = r_next;
      r_next = r_after;
      r_after = roles_of(i + 2);
      uint32_t m4 = 0, c4 = 0;
      uint32_t ent[4] = {0u, 0u, 0u, 0u};
      uint32_t kk[4] = {0u, 0u, 0u, 0u};
      if (g < ngroups) {
        const uint4 kv = kv_of(g);
        kk[0] = kv.x;
        kk[1] = kv.y;
        kk[2] = kv.z;
        kk[3] = kv.w;
        const uint32_t fb = floor_bits(4 * g - off, v.nf, n);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t r = (rw >> (8 * j)) & 0xFFu;
          const int T = S.first_of_role[r];
          const int hb = static_cast<int>(kk[j] >> shd);
          m4 |= static_cast<uint32_t>(hb > T) << j;
          if (hb == T && !((fb >> j) & 1u)) {
            c4 |= 1u << j;
            ent[j] = (static_cast<uint32_t>(S.code_of_role[r]) << (STREAM ? 24 : 16)) |
                     static_cast<uint32_t>(4 * g + j);
          }
        }
        m4 |= fb;                                  // the recency floor is kept
      }
      store_bits(bits, g, nwords, lane, m4);
      // list slots: lane's rank among the warp's candidates from four ballots
      const int nc = __popc(c4);
      const unsigned b1 = __ballot_sync(0xffffffffu, nc >= 1);
      if (b1 != 0) {
        const unsigned b2 = __ballot_sync(0xffffffffu, nc >= 2);
        const unsigned b3 = __ballot_sync(0xffffffffu, nc >= 3);
        const unsigned b4 = __ballot_sync(0xffffffffu, nc >= 4);
        const unsigned lt = (1u << lane) - 1u;
        int base = 0;
        if (lane == 0) base = atomicAdd(&S.list_n, __popc(b1) + __popc(b2) + __popc(b3) + __popc(b4));
        base = __shfl_sync(0xffffffffu, base, 0);
        int pos = base + __popc(b1 & lt) + __popc(b2 & lt) + __popc(b3 & lt) + __popc(b4 & lt);
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if ((c4 >> j) & 1u) {
            if (pos < list_cap) {
              if (STREAM) {
                list[2 * pos] = kk[j];
                list[2 * pos + 1] = ent[j];
              } else {
                list[pos] = ent[j];
              }
            }
            ++pos;
          }
      }
    }
    __syncthreads();
    if (S.list_n > list_cap) {
      if (tid == 0) S.general = 1;   // (cannot happen: the counts bound the list)
      __syncthreads();
    }
  }

  if (!S.general) {
    if (any_thr) {
      // ---- remaining bits over the candidate list
      const int m = S.list_n;
      for (int lo = shd; lo > 0;) {
        const int d = lo < 8 ? lo : 8;
        const int shift = lo - d;
        for (int e = tid; e < m; e += NT) {
          const uint32_t ent = STREAM ? list[2 * e + 1] : list[e];
          const uint32_t c = STREAM ? ent >> 24 : ent >> 16;
          const uint32_t key = STREAM ? list[2 * e] : keys[ent & 0xFFFFu];
          if ((key >> lo) == (S.prefix[c] >> lo))
            atomicAdd(&S.hist[c][(key >> shift) & ((1u << d) - 1u)], 1);
        }
        __syncthreads();
        if (warp < kR && S.mode[warp] == 2) descend(S, warp, lane, shift);
        __syncthreads();
        lo = shift;
      }
      // kept candidates join the bits; ties of partial buckets are gathered
      const uint32_t partial = S.partial_ties;
      for (int e = tid; e < m; e += NT) {
        const uint32_t ent = STREAM ? list[2 * e + 1] : list[e];
        const uint32_t c = STREAM ? ent >> 24 : ent >> 16;
        const uint32_t slot = STREAM ? ent & 0xFFFFFFu : ent & 0xFFFFu;
        const uint32_t key = STREAM ? list[2 * e] : keys[slot];
        if (key >= S.thr[c]) {
          atomicOr(&bits[slot >> 5], 1u << (slot & 31u));
        } else if (((partial >> c) & 1u) && key == S.prefix[c]) {
          const int t = atomicAdd(&S.tie_n, 1);
          if (t < kTieCap) S.ties[t] = ent;
        }
      }
      __syncthreads();
      const int nt = S.tie_n;
      if (partial != 0 && nt <= kTieCap) {
        // index-order rank among the bucket's ties
        constexpr int kCodeShift = STREAM ? 24 : 16;
        constexpr uint32_t kSlotMask = STREAM ? 0xFFFFFFu : 0xFFFFu;
        for (int t = tid; t < nt; t += NT) {
          const uint32_t ent = S.ties[t];
          const uint32_t c = ent >> kCodeShift, slot = ent & kSlotMask;
          int rank = 0;
          for (int x = 0; x < nt; ++x) {
            const uint32_t o = S.ties[x];
            rank += ((o >> kCodeShift) == c && (o & kSlotMask) < slot);
          }
          if (rank < S.need[c]) atomicOr(&bits[slot >> 5], 1u << (slot & 31u));
        }
        __syncthreads();
      } else if (partial != 0) {
        if (tid == 0) S.general = 2;   // too many ties: rank them over all slots
        __syncthreads();
      }
    }
  } else {
    // ---- general path: four 8-bit rounds over every slot, from the top
    // (the first-digit step may have run before the list overflowed)
    if (tid < kR) {
      S.prefix[tid] = 0;
      S.need[tid] = S.quota[tid];
    }
    __syncthreads();
    for (int round = 0; round < (any_thr ? 4 : 0); ++round) {
      const int shift = 24 - 8 * round;
      for (int i = 0; i < iters; ++i) {
        const int g = i * NT + tid;
        if (g >= ngroups) break;
        const uint4 kv = kv_of(g);
        const uint32_t kk[4] = {kv.x, kv.y, kv.z, kv.w};
        const uint32_t rw = load_roles(v.rp, off, n, g, v.rvec);
        const uint32_t fb = floor_bits(4 * g - off, v.nf, n);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t c = static_cast<uint32_t>(S.code_of_role[(rw >> (8 * j)) & 0xFFu]);
          if (c >= static_cast<uint32_t>(kR) || ((fb >> j) & 1u)) continue;
          if (round > 0 && (kk[j] >> (shift + 8)) != (S.prefix[c] >> (shift + 8))) continue;
          atomicAdd(&S.hist[c][(kk[j] >> shift) & 0xFFu], 1);
        }
      }
      __syncthreads();
      if (warp < kR && S.mode[warp] == 2) descend(S, warp, lane, shift);
      __syncthreads();
    }
    for (int i = 0; i < iters; ++i) {
      const int g = i * NT + tid;
      uint32_t m4 = 0;
      if (g < ngroups) {
        const uint4 kv = kv_of(g);
        const uint32_t kk[4] = {kv.x, kv.y, kv.z, kv.w};
        const uint32_t rw = load_roles(v.rp, off, n, g, v.rvec);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t c = static_cast<uint32_t>(S.code_of_role[(rw >> (8 * j)) & 0xFFu]);
          const bool keep = (c < static_cast<uint32_t>(kR)) ? (kk[j] >= S.thr[c]) : (c == kCodeKeep);
          m4 |= static_cast<uint32_t>(keep) << j;
        }
        m4 |= floor_bits(4 * g - off, v.nf, n);    // the recency floor is kept
      }
      store_bits(bits, g, nwords, lane, m4);
    }
    __syncthreads();
  }

  // Ties beyond the shared-memory list (general path, or too many ties): the
  // first need[b] keys equal to the threshold, in index order, over all slots.
  if (S.general) {
    for (uint32_t pend = S.partial_ties; pend != 0; pend &= pend - 1) {
      const int b = __ffs(pend) - 1;
      const uint32_t P = S.prefix[b];
      const int need = S.need[b];
      auto tie_mask = [&](int q) {
        uint32_t mk = 0;
#pragma unroll
        for (int gg = 0; gg < 8; ++gg) {
          const int g = 8 * q + gg;
          if (g >= ngroups) break;
          const uint4 kv = kv_of(g);
          const uint32_t kk[4] = {kv.x, kv.y, kv.z, kv.w};
          const uint32_t rw = load_roles(v.rp, off, n, g, v.rvec);
          const uint32_t fb = floor_bits(4 * g - off, v.nf, n);
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (S.code_of_role[(rw >> (8 * j)) & 0xFFu] == b && kk[j] == P && !((fb >> j) & 1u))
              mk |= 1u << (4 * gg + j);
        }
        return mk;
      };
      scan_words<NT>(nwords, tie_mask, [&](int q, uint32_t mk, int rank) {
        uint32_t keepm = 0;
        while (mk != 0 && rank < need) {
          const uint32_t low = mk & (0u - mk);
          keepm |= low;
          mk ^= low;
          ++rank;
        }
        if (keepm) bits[q] |= keepm;
      }, S.warp_tot);
    }
  }

  // ---- SLACK: the slots saturated buckets left go to the best-scoring
  // tokens of eligible roles not kept yet (ties to the lower index).  With
  // the fill's first digit known (sfast), one pass keeps such tokens above
  // it and lists those at it; the remaining bits are resolved over the list
  // in the state of bucket 0, whose own selection is complete.
  if (!STREAM && S.slack > 0 && S.sfast) {
    const uint32_t elig = S.elig_mask;
    const int sh0 = 31 - nb;
    const uint32_t bmask = (1u << nb) - 1u;
    const uint32_t DS = (S.sprefix >> sh0) & bmask;
    if (tid == 0) {
      S.list_n = 0;
      S.tie_n = 0;
      S.partial_ties = 0;
      S.prefix[0] = S.sprefix;
      S.need[0] = S.sneed;
      S.thr[0] = 0xFFFFFFFFu;
    }
    for (int x = tid; x < 256; x += NT) S.hist[0][x] = 0;
    __syncthreads();
    for (int i = 0; i < iters; ++i) {
      const int g = i * NT + tid;
      uint32_t m4 = 0, c4 = 0;
      if (g < ngroups) {
        const uint4 kv = keys4[g];
        const uint32_t kk[4] = {kv.x, kv.y, kv.z, kv.w};
        const uint32_t rw = load_roles(v.rp, off, n, g, v.rvec);
        const uint32_t fb = floor_bits(4 * g - off, v.nf, n);
        const uint32_t kb = (bits[g >> 3] >> (4 * (g & 7))) & 0xFu;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint32_t r = (rw >> (8 * j)) & 0xFFu;
          if (r >= static_cast<uint32_t>(kR) || !((elig >> r) & 1u) || ((fb | kb) >> j) & 1u) continue;
          const uint32_t d = (kk[j] >> sh0) & bmask;
          m4 |= static_cast<uint32_t>(d > DS) << j;
          c4 |= static_cast<uint32_t>(d == DS) << j;
        }
        if (m4) atomicOr(&bits[g >> 3], m4 << (4 * (g & 7)));
      }
      const int nc = __popc(c4);
      const unsigned b1 = __ballot_sync(0xffffffffu, nc >= 1);
      if (b1 != 0) {
        const unsigned b2 = __ballot_sync(0xffffffffu, nc >= 2);
        const unsigned b3 = __ballot_sync(0xffffffffu, nc >= 3);
        const unsigned b4 = __ballot_sync(0xffffffffu, nc >= 4);
        const unsigned lt = (1u << lane) - 1u;
        int base = 0;
        if (lane == 0) base = atomicAdd(&S.list_n, __popc(b1) + __popc(b2) + __popc(b3) + __popc(b4));
        base = __shfl_sync(0xffffffffu, base, 0);
        int pos = base + __popc(b1 & lt) + __popc(b2 & lt) + __popc(b3 & lt) + __popc(b4 & lt);
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if ((c4 >> j) & 1u) {
            if (pos < list_cap) list[pos] = static_cast<uint32_t>(4 * g + j);
            ++pos;
          }
      }
    }
    __syncthreads();
    // (the histograms bound the listed count by list_cap)
    const int m = S.list_n < list_cap ? S.list_n : list_cap;
    for (int lo = sh0; lo > 0;) {
      const int d = lo < 8 ? lo : 8;
      const int shift = lo - d;
      for (int e = tid; e < m; e += NT) {
        const uint32_t key = keys[list[e]];
        if ((key >> lo) == (S.prefix[0] >> lo)) atomicAdd(&S.hist[0][(key >> shift) & ((1u << d) - 1u)], 1);
      }
      __syncthreads();
      if (warp == 0) descend(S, 0, lane, shift);
      __syncthreads();
      lo = shift;
    }
    const uint32_t T = S.thr[0], P = S.prefix[0];
    const int need = S.need[0];
    const bool partial = S.partial_ties & 1u;
    for (int e = tid; e < m; e += NT) {
      const uint32_t slot = list[e];
      const uint32_t key = keys[slot];
      if (key >= T) {
        atomicOr(&bits[slot >> 5], 1u << (slot & 31u));
      } else if (partial && key == P) {
        const int t = atomicAdd(&S.tie_n, 1);
        if (t < kTieCap) S.ties[t] = slot;
      }
    }
    __syncthreads();
    const int nt = S.tie_n;
    if (partial && nt <= kTieCap) {
      // index-order rank among the fill's ties
      for (int t = tid; t < nt; t += NT) {
        const uint32_t slot = S.ties[t];
        int rank = 0;
        for (int x = 0; x < nt; ++x) rank += S.ties[x] < slot;
        if (rank < need) atomicOr(&bits[slot >> 5], 1u << (slot & 31u));
      }
      __syncthreads();
    } else if (partial) {
      // more ties than the shared list holds: rank them over all slots
      auto tie_mask = [&](int q) {
        uint32_t mk = 0;
#pragma unroll
        for (int gg = 0; gg < 8; ++gg) {
          const int g = 8 * q + gg;
          if (g >= ngroups) break;
          const uint4 kv = keys4[g];
          const uint32_t kk[4] = {kv.x, kv.y, kv.z, kv.w};
          const uint32_t rw = load_roles(v.rp, off, n, g, v.rvec);
          const uint32_t fb = floor_bits(4 * g - off, v.nf, n);
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const uint32_t r = (rw >> (8 * j)) & 0xFFu;
            const int slot = 4 * g + j;
            if (kk[j] == P && r < static_cast<uint32_t>(kR) && ((elig >> r) & 1u) && !((fb >> j) & 1u) &&
                !((bits[slot >> 5] >> (slot & 31)) & 1u))
              mk |= 1u << (4 * gg + j);
          }
        }
        return mk;
      };
      scan_words<NT>(nwords, tie_mask, [&](int q, uint32_t mk, int rank) {
        uint32_t keepm = 0;
        while (mk != 0 && rank < need) {
          const uint32_t low = mk & (0u - mk);
          keepm |= low;
          mk ^= low;
          ++rank;
        }
        if (keepm) bits[q] |= keepm;
      }, S.warp_tot);
    }
  } else if (S.slack > 0) {
    const uint32_t elig = S.elig_mask;
    auto candidate = [&](uint32_t rw, uint32_t fb, int g, int j) {
      const uint32_t r = (rw >> (8 * j)) & 0xFFu;
      const int slot = 4 * g + j;
      return r < static_cast<uint32_t>(kR) && ((elig >> r) & 1u) && !((fb >> j) & 1u) &&
             !((bits[slot >> 5] >> (slot & 31)) & 1u);
    };
    if (tid == 0) {
      S.prefix[0] = 0;
      S.need[0] = S.slack;
      S.partial_ties = 0;
    }
    for (int x = tid; x < 256; x += NT) S.hist[0][x] = 0;
    __syncthreads();
    for (int round = 0; round < 4; ++round) {
      const int shift = 24 - 8 * round;
      for (int i = 0; i < iters; ++i) {
        const int g = i * NT + tid;
        if (g >= ngroups) break;
        const uint4 kv = kv_of(g);
        const uint32_t kk[4] = {kv.x, kv.y, kv.z, kv.w};
        const uint32_t rw = load_roles(v.rp, off, n, g, v.rvec);
        const uint32_t fb = floor_bits(4 * g - off, v.nf, n);
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          if (!candidate(rw, fb, g, j)) continue;
          if (round > 0 && (kk[j] >> (shift + 8)) != (S.prefix[0] >> (shift + 8))) continue;
          atomicAdd(&S.hist[0][(kk[j] >> shift) & 0xFFu], 1);
        }
      }
      __syncthreads();
      if (warp == 0) descend(S, 0, lane, shift);
      __syncthreads();
    }
    // candidates above the threshold join; the rest of the ties in index order
    const uint32_t T = S.thr[0], P = S.prefix[0];
    const int need = S.need[0];
    const bool partial = S.partial_ties & 1u;
    __syncthreads();
    for (int i = 0; i < iters; ++i) {
      const int g = i * NT + tid;
      if (g >= ngroups) break;
      const uint4 kv = kv_of(g);
      const uint32_t kk[4] = {kv.x, kv.y, kv.z, kv.w};
      const uint32_t rw = load_roles(v.rp, off, n, g, v.rvec);
      const uint32_t fb = floor_bits(4 * g - off, v.nf, n);
      uint32_t m4 = 0;
#pragma unroll
      for (int j = 0; j < 4; ++j)
        if (kk[j] >= T && candidate(rw, fb, g, j)) m4 |= 1u << j;
      if (m4) atomicOr(&bits[g >> 3], m4 << (4 * (g & 7)));
    }
    __syncthreads();
    if (partial) {
      auto tie_mask = [&](int q) {
        uint32_t mk = 0;
#pragma unroll
        for (int gg = 0; gg < 8; ++gg) {
          const int g = 8 * q + gg;
          if (g >= ngroups) break;
          const uint4 kv = kv_of(g);
          const uint32_t kk[4] = {kv.x, kv.y, kv.z, kv.w};
          const uint32_t rw = load_roles(v.rp, off, n, g, v.rvec);
          const uint32_t fb = floor_bits(4 * g - off, v.nf, n);
#pragma unroll
          for (int j = 0; j < 4; ++j)
            if (kk[j] == P && candidate(rw, fb, g, j)) mk |= 1u << (4 * gg + j);
        }
        return mk;
      };
      scan_words<NT>(nwords, tie_mask, [&](int q, uint32_t mk, int rank) {
        uint32_t keepm = 0;
        while (mk != 0 && rank < need) {
          const uint32_t low = mk & (0u - mk);
          keepm |= low;
          mk ^= low;
          ++rank;
        }
        if (keepm) bits[q] |= keepm;
      }, S.warp_tot);
    }
  }

  // ---- kept positions in ascending order
  int32_t* dst = a.keep_idx + S.keep_off;
  const bool count_roles = a.kept_per_role != nullptr &&
                           (a.policy == ROLEKV_POLICY_GLOBAL || a.policy == ROLEKV_POLICY_SLACK);
  uint64_t kr = 0;
  const int total = scan_words<NT>(nwords, [&](int q) { return bits[q]; }, [&](int q, uint32_t m, int pos) {
    while (m != 0) {
      const int t = q * 32 + (__ffs(m) - 1) - off;
      m &= m - 1;
      if (in_bounds(pos, 1, width, a.status)) dst[pos] = t;   // (the unit's own row)
      ++pos;
      if (count_roles) kr += shl64(1ull, 8u * __ldg(v.rp + t));
    }
  }, S.warp_tot);
  for (int64_t j = total + tid; j < width; j += NT) dst[j] = -1;

  if (a.keep_mask != nullptr) {
    uint8_t* mp = a.keep_mask + sbase;
    const bool mvec = ((reinterpret_cast<uintptr_t>(mp) - static_cast<uintptr_t>(off)) & 3u) == 0;
    for (int g = tid; g < ngroups; g += NT) {
      const uint32_t m4 = (bits[g >> 3] >> (4 * (g & 7))) & 15u;
      const int s0 = 4 * g - off;
      if (mvec && s0 >= 0 && s0 + 4 <= n) {
        const uint32_t w = (m4 & 1u) | ((m4 >> 1) & 1u) << 8 | ((m4 >> 2) & 1u) << 16 | ((m4 >> 3) & 1u) << 24;
        *reinterpret_cast<uint32_t*>(mp + s0) = w;
      } else {
#pragma unroll
        for (int j = 0; j < 4; ++j)
          if (s0 + j >= 0 && s0 + j < n) mp[s0 + j] = static_cast<uint8_t>((m4 >> j) & 1u);
      }
    }
  }

  if (a.kept_per_role != nullptr) {
    if (count_roles) {
#pragma unroll
      for (int r = 0; r < kR; ++r) {
        const int c = warp_sum(static_cast<int>((kr >> (8 * r)) & 0xFFu));
        if (lane == 0 && c) atomicAdd(&S.kept_role[r], c);
      }
      __syncthreads();
    }
    if (tid < a.n_roles)
      a.kept_per_role[static_cast<int64_t>(u) * a.n_roles + tid] =
          count_roles ? S.kept_role[tid] : S.quota[tid] + S.floor_role[tid];
  }
  if (tid == 0 && S.nan_seen && a.status != nullptr) atomicOr(a.status, ROLEKV_STATUS_NONFINITE);
}

template <int NT, bool STREAM>
cudaError_t launch_select_nt(const SelectArgs& a, size_t smem, cudaStream_t stream) {
  cudaError_t e = cudaFuncSetAttribute(select_kernel<NT, STREAM>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  select_kernel<NT, STREAM><<<a.n_units, NT, smem, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace

size_t select_smem_bytes(int n_max) {
  const size_t groups = static_cast<size_t>(select_groups(n_max));
  return (n_max > kSmemMaxN ? 0 : groups * 16) + groups / 8 * 4 + region_bytes(n_max);
}

cudaError_t launch_select(const SelectArgs& a, cudaStream_t stream) {
  if (a.n_units == 0) return cudaSuccess;
  const size_t smem = select_smem_bytes(a.n_max);
  // CTA size follows the row length so that short rows still fill the SM
  // with several CTAs (shared memory is sized by the longest row).
  if (a.n_max > kSmemMaxN) return launch_select_nt<1024, true>(a, smem, stream);
  if (a.n_max > 16384) return launch_select_nt<1024, false>(a, smem, stream);
  if (a.n_max > 8192) return launch_select_nt<512, false>(a, smem, stream);
  return launch_select_nt<256, false>(a, smem, stream);
}

}  // namespace rolekv
