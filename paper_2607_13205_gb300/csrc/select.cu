// Role-conditional allocation and per-bucket top-k (Section 4.1, Algorithm 1):
// pool the scores (optional), count the roles, split the budget ceil(B n)
// across role buckets, and keep the top-q_r tokens of every bucket, ties to the
// lower index.  One CTA per (layer, sequence, KV head) holds the whole score
// row in shared memory; everything after the fp32 -> ordered-key mapping is
// integer, so the kept set is bit-exact for a given score row.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "device_common.cuh"
#include "internal.h"

namespace rolekv {
namespace {

constexpr int kThreads = 1024;
constexpr int kWarps = kThreads / 32;
constexpr int kMaxPerThread = (ROLEKV_SELECT_MAX_N + kThreads - 1) / kThreads;
constexpr int kR = ROLEKV_MAX_ROLES;

// Monotone map of a float to uint32 (larger float -> larger key); -0 is folded
// onto +0 so equal floats give equal keys.
__device__ __forceinline__ uint32_t ordered_key(float f) {
  if (f == 0.0f) f = 0.0f;
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

struct SelShared {
  int64_t quota[kR];
  int64_t size[kR];
  int32_t bucket_of_role[256];
  uint32_t prefix[kR];
  uint32_t need[kR];
  int32_t mode[kR];              // 0 none kept, 1 all kept, 2 threshold
  int32_t hist[kR][256];
  int32_t warp_cnt[kWarps][kR];  // per-warp tie counts, then exclusive bases
  int32_t warp_kept[kWarps];
  int32_t kept_role[kR];
  int64_t keep_off;
  int32_t nonfinite;
};

__device__ __forceinline__ int warp_sum(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Integer quotas of one sequence; the same arithmetic as the public
// description in rolekv.h (water-filling then largest remainder).
__device__ void compute_quotas(const SelectArgs& a, const int64_t* count, int64_t K_full,
                               int64_t* q) {
  for (int r = 0; r < kR; ++r) q[r] = 0;
  const int R = a.n_roles;
  if (a.policy == ROLEKV_POLICY_GLOBAL) {
    int64_t elig = 0;
    for (int r = 0; r < R; ++r)
      if (!((a.ban_mask >> r) & 1u)) elig += count[r];
    q[0] = K_full < elig ? K_full : elig;
    return;
  }
  bool live[kR];
  int64_t elig = 0;
  for (int r = 0; r < kR; ++r) {
    live[r] = (r < R) && a.alpha_fx[r] > 0 && count[r] > 0;
    if (live[r]) elig += count[r];
  }
  const int64_t K = K_full < elig ? K_full : elig;
  int64_t left = K;
  bool changed = true;
  while (changed) {
    changed = false;
    int64_t A = 0;
    for (int r = 0; r < kR; ++r)
      if (live[r]) A += a.alpha_fx[r];
    if (A == 0) break;
    bool sat[kR];
    for (int r = 0; r < kR; ++r) sat[r] = live[r] && a.alpha_fx[r] * left >= count[r] * A;
    for (int r = 0; r < kR; ++r)
      if (sat[r]) {
        q[r] = count[r];
        live[r] = false;
        changed = true;
      }
    for (int r = 0; r < kR; ++r)
      if (sat[r]) left -= count[r];
  }
  int64_t A = 0;
  for (int r = 0; r < kR; ++r)
    if (live[r]) A += a.alpha_fx[r];
  if (A == 0) return;
  int64_t rem[kR];
  int64_t given = 0;
  for (int r = 0; r < kR; ++r)
    if (live[r]) {
      q[r] = (a.alpha_fx[r] * left) / A;
      rem[r] = (a.alpha_fx[r] * left) % A;
      given += q[r];
    }
  int64_t extra = left - given;
  while (extra > 0) {
    int best = -1;
    for (int r = 0; r < kR; ++r)
      if (live[r] && (best < 0 || rem[r] > rem[best])) best = r;
    q[best] += 1;
    live[best] = false;
    --extra;
  }
}

__global__ void __launch_bounds__(kThreads, 1) select_kernel(const SelectArgs a) {
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
  const int64_t K_s = kept_slots(n, a.budget_fx);

  uint32_t* keys = reinterpret_cast<uint32_t*>(dyn);
  uint8_t* roles = dyn + static_cast<size_t>(a.n_max) * 4;
  uint32_t* keptbits = reinterpret_cast<uint32_t*>(roles + ((a.n_max + 15) & ~15));

  // ---- offsets of this unit's kept row
  if (tid < kR) {
    S.kept_role[tid] = 0;
  }
  if (tid == 0) S.nonfinite = 0;
  {
    int64_t part = 0;
    if (a.varlen) {
      for (int x = tid; x < s; x += kThreads)
        part += kept_slots(a.cu_seqlens[x + 1] - a.cu_seqlens[x], a.budget_fx);
    }
    // block reduction of `part` through the warp_kept scratch
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
    __shared__ int64_t red64[kWarps];
    if (lane == 0) red64[warp] = part;
    __syncthreads();
    if (tid == 0) {
      int64_t cu = 0;
      for (int w = 0; w < kWarps; ++w) cu += red64[w];
      S.keep_off = a.varlen ? (static_cast<int64_t>(l) * a.Hkv + h) * a.Ktot + cu
                            : static_cast<int64_t>(u) * a.K_dense;
    }
  }

  // ---- load roles and scores, pool, map to ordered keys
  for (int t = tid; t < n; t += kThreads) roles[t] = a.roles[rbase + t];
  if (a.pool_k <= 1) {
    for (int t = tid; t < n; t += kThreads) {
      const float f = a.scores[sbase + t];
      if (isnan(f)) S.nonfinite = 1;
      keys[t] = isnan(f) ? 0u : ordered_key(f);
    }
  } else {
    for (int t = tid; t < n; t += kThreads) keys[t] = __float_as_uint(a.scores[sbase + t]);
    __syncthreads();
    float pooled[kMaxPerThread];
    const int hw = a.pool_k / 2;
#pragma unroll
    for (int i = 0; i < kMaxPerThread; ++i) {
      const int t = tid + i * kThreads;
      float m = 0.f;
      if (t < n) {
        const int lo = max(0, t - hw), hi = min(n - 1, t + hw);
        m = __uint_as_float(keys[lo]);
        bool nan_seen = isnan(m);
        for (int x = lo + 1; x <= hi; ++x) {
          const float v = __uint_as_float(keys[x]);
          nan_seen |= isnan(v);
          m = fmaxf(m, v);
        }
        if (nan_seen) {
          S.nonfinite = 1;
          m = NAN;
        }
      }
      pooled[i] = m;
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < kMaxPerThread; ++i) {
      const int t = tid + i * kThreads;
      if (t < n) keys[t] = isnan(pooled[i]) ? 0u : ordered_key(pooled[i]);
    }
  }

  // ---- role counts
  {
    int cnt[kR];
#pragma unroll
    for (int r = 0; r < kR; ++r) cnt[r] = 0;
    for (int t = tid; t < n; t += kThreads) {
      const int r = roles[t];
#pragma unroll
      for (int x = 0; x < kR; ++x) cnt[x] += (r == x);
    }
    if (tid < kR) S.size[tid] = 0;
    __syncthreads();
#pragma unroll
    for (int r = 0; r < kR; ++r) {
      const int v = warp_sum(cnt[r]);
      if (lane == 0 && v) atomicAdd(reinterpret_cast<unsigned long long*>(&S.size[r]),
                                    static_cast<unsigned long long>(v));
    }
    __syncthreads();
  }

  // ---- quotas and bucket sizes
  if (tid == 0) {
    int64_t count[kR];
    for (int r = 0; r < kR; ++r) count[r] = (r < a.n_roles) ? S.size[r] : 0;
    int64_t q[kR];
    compute_quotas(a, count, K_s, q);
    int64_t bsize[kR];
    for (int r = 0; r < kR; ++r) bsize[r] = 0;
    if (a.policy == ROLEKV_POLICY_GLOBAL) {
      for (int r = 0; r < a.n_roles; ++r)
        if (!((a.ban_mask >> r) & 1u)) bsize[0] += count[r];
    } else {
      for (int r = 0; r < kR; ++r) bsize[r] = count[r];
    }
    for (int r = 0; r < kR; ++r) {
      S.quota[r] = q[r];
      S.size[r] = bsize[r];
      S.mode[r] = (q[r] <= 0) ? 0 : (q[r] >= bsize[r] ? 1 : 2);
      S.prefix[r] = 0;
      S.need[r] = static_cast<uint32_t>(q[r]);
    }
  }
  for (int x = tid; x < 256; x += kThreads) {
    int b = -1;
    if (x < a.n_roles && !((a.ban_mask >> x) & 1u))
      b = (a.policy == ROLEKV_POLICY_GLOBAL) ? 0 : x;
    S.bucket_of_role[x] = b;
  }
  __syncthreads();

  // ---- radix threshold per bucket: 4 rounds of 8-bit digits, most
  // significant first; after them prefix[b] is the q_b-th largest key of the
  // bucket and need[b] the number of tokens equal to it that are kept.
  bool any_threshold = false;
#pragma unroll
  for (int r = 0; r < kR; ++r) any_threshold |= (S.mode[r] == 2);
  if (any_threshold) {
    for (int round = 0; round < 4; ++round) {
      const int shift = 24 - 8 * round;
      const uint32_t hi_mask = (round == 0) ? 0u : (0xFFFFFFFFu << (shift + 8));
      for (int x = tid; x < kR * 256; x += kThreads) (&S.hist[0][0])[x] = 0;
      __syncthreads();
      const int steps = (n + kThreads - 1) / kThreads;
      for (int st = 0; st < steps; ++st) {
        const int t = st * kThreads + tid;
        int b = -1;
        uint32_t key = 0;
        if (t < n) {
          b = S.bucket_of_role[roles[t]];
          key = keys[t];
          if (b >= 0 && (S.mode[b] != 2 || (key & hi_mask) != S.prefix[b])) b = -1;
        }
        const int digit = (key >> shift) & 255;
        const int tag = (b < 0) ? -1 : (b << 8) | digit;
        const unsigned peers = __match_any_sync(0xffffffffu, tag);
        if (tag >= 0 && (__ffs(peers) - 1) == lane)
          atomicAdd(&S.hist[b][digit], __popc(peers));
      }
      __syncthreads();
      if (warp < kR && S.mode[warp] == 2) {
        const int b = warp;
        // lane handles digits [lane*8, lane*8+8); suffix sums from the top
        int c[8];
        int mine = 0;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          c[i] = S.hist[b][lane * 8 + i];
          mine += c[i];
        }
        // above = tokens whose digit falls in a higher lane's range
        int incl = mine;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int v = __shfl_down_sync(0xffffffffu, incl, o);
          if (lane + o < 32) incl += v;
        }
        const int above = incl - mine;
        const int need = static_cast<int>(S.need[b]);
        // the digit where the count of larger-or-equal keys first reaches need
        int found_digit = -1, gt_before = 0;
        if (above < need && above + mine >= need) {
          int acc = above;
          for (int i = 7; i >= 0; --i) {
            if (acc + c[i] >= need) {
              found_digit = lane * 8 + i;
              gt_before = acc;
              break;
            }
            acc += c[i];
          }
        }
        const unsigned who = __ballot_sync(0xffffffffu, found_digit >= 0);
        const int src = who ? __ffs(who) - 1 : 0;
        const int fd = __shfl_sync(0xffffffffu, found_digit, src);
        const int gb = __shfl_sync(0xffffffffu, gt_before, src);
        if (lane == 0 && who != 0) {
          S.prefix[b] |= static_cast<uint32_t>(fd) << shift;
          S.need[b] = static_cast<uint32_t>(need - gb);
        }
      }
      __syncthreads();
    }
  }

  // ---- tie ranks in index order and the kept set.  Warp w owns the token
  // range [w*seg, (w+1)*seg).
  const int seg = ((n + kWarps - 1) / kWarps + 31) & ~31;
  const int t_begin = warp * seg;
  const int t_end = min(n, t_begin + seg);
  const unsigned lt_mask = (1u << lane) - 1u;
  // pass A: ties per bucket in this warp's range
  {
    int tie_cnt[kR];
#pragma unroll
    for (int r = 0; r < kR; ++r) tie_cnt[r] = 0;
    for (int t0 = t_begin; t0 < t_end; t0 += 32) {
      const int t = t0 + lane;
      int b = -1;
      if (t < t_end) {
        b = S.bucket_of_role[roles[t]];
        if (b >= 0 && !(S.mode[b] == 2 && keys[t] == S.prefix[b])) b = -1;
      }
#pragma unroll
      for (int r = 0; r < kR; ++r) tie_cnt[r] += __popc(__ballot_sync(0xffffffffu, b == r));
    }
    if (lane < kR) {
      int v = 0;
#pragma unroll
      for (int r = 0; r < kR; ++r) v = (lane == r) ? tie_cnt[r] : v;
      S.warp_cnt[warp][lane] = v;
    }
  }
  __syncthreads();
  if (tid < kR) {   // exclusive scan over warps, bucket `tid`
    int run = 0;
    for (int w = 0; w < kWarps; ++w) {
      const int v = S.warp_cnt[w][tid];
      S.warp_cnt[w][tid] = run;
      run += v;
    }
  }
  __syncthreads();
  // pass B: decide, record bits, count per warp and per role
  {
    int tie_run[kR];
#pragma unroll
    for (int r = 0; r < kR; ++r) tie_run[r] = S.warp_cnt[warp][r];
    int kept_here = 0;
    int role_kept[kR];
#pragma unroll
    for (int r = 0; r < kR; ++r) role_kept[r] = 0;
    for (int t0 = t_begin; t0 < t_end; t0 += 32) {
      const int t = t0 + lane;
      bool keep = false;
      int b = -1, tie_b = -1, role = 0;
      if (t < t_end) {
        role = roles[t];
        b = S.bucket_of_role[role];
        if (b >= 0) {
          const int md = S.mode[b];
          if (md == 1) {
            keep = true;
          } else if (md == 2) {
            const uint32_t k = keys[t];
            if (k > S.prefix[b]) keep = true;
            else if (k == S.prefix[b]) tie_b = b;
          }
        }
      }
#pragma unroll
      for (int r = 0; r < kR; ++r) {
        const unsigned m = __ballot_sync(0xffffffffu, tie_b == r);
        if (tie_b == r) keep = (tie_run[r] + __popc(m & lt_mask)) < static_cast<int>(S.need[r]);
        tie_run[r] += __popc(m);
      }
      const unsigned km = __ballot_sync(0xffffffffu, keep);
      if (lane == 0 && t0 < t_end) {
        // bits of tokens t0 .. t0+31 (t0 is a multiple of 32)
        keptbits[t0 >> 5] = km;
      }
      kept_here += __popc(km);
      if (keep) {
#pragma unroll
        for (int r = 0; r < kR; ++r) role_kept[r] += (role == r);
      }
      if (a.keep_mask != nullptr && t < t_end) a.keep_mask[sbase + t] = keep ? 1 : 0;
    }
    if (lane == 0) S.warp_kept[warp] = kept_here;
    if (a.kept_per_role != nullptr) {
#pragma unroll
      for (int r = 0; r < kR; ++r) {
        const int v = warp_sum(role_kept[r]);
        if (lane == 0 && v) atomicAdd(&S.kept_role[r], v);
      }
    }
  }
  __syncthreads();
  if (tid == 0) {
    int run = 0;
    for (int w = 0; w < kWarps; ++w) {
      const int v = S.warp_kept[w];
      S.warp_kept[w] = run;
      run += v;
    }
    S.warp_cnt[0][0] = run;   // total kept (the scan above is no longer needed)
  }
  __syncthreads();
  // pass C: write kept positions in ascending order
  {
    int out = S.warp_kept[warp];
    int32_t* dst = a.keep_idx + S.keep_off;
    for (int t0 = t_begin; t0 < t_end; t0 += 32) {
      const unsigned km = keptbits[t0 >> 5];
      if ((km >> lane) & 1u) dst[out + __popc(km & lt_mask)] = t0 + lane;
      out += __popc(km);
    }
    const int total = S.warp_cnt[0][0];
    for (int64_t j = total + tid; j < K_s; j += kThreads) dst[j] = -1;
  }
  if (a.kept_per_role != nullptr && tid < a.n_roles)
    a.kept_per_role[static_cast<int64_t>(u) * a.n_roles + tid] = S.kept_role[tid];
  if (tid == 0 && S.nonfinite && a.status != nullptr) atomicOr(a.status, ROLEKV_STATUS_NONFINITE);
}

}  // namespace

size_t select_smem_bytes(int n_max) {
  const size_t keys = static_cast<size_t>(n_max) * 4;
  const size_t roles = (static_cast<size_t>(n_max) + 15) & ~static_cast<size_t>(15);
  const size_t bits = ((static_cast<size_t>(n_max) + 31) / 32 + 32) * 4;
  return keys + roles + bits;
}

cudaError_t launch_select(const SelectArgs& a, cudaStream_t stream) {
  if (a.n_units == 0) return cudaSuccess;
  const size_t smem = select_smem_bytes(a.n_max);
  cudaError_t e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  select_kernel<<<a.n_units, kThreads, smem, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace rolekv
