// Quest one-shot analogue (Section 5, "Query-aware baseline"): the mean
// query of the SnapKV window scores every page of `page` consecutive keys by
// Quest's key bound, sum_i max(qbar_i * min_t k_ti, qbar_i * max_t k_ti), an
// upper bound on qbar . k_t for every token t of the page; every token gets
// its page's bound, so the role-conditional selector (or its GLOBAL top-k)
// runs on it unchanged.  One CTA per (layer, sequence, KV head): the mean of
// the G x W_eff window rows goes to shared memory, then each warp takes whole
// pages, streaming their key rows with 16-byte read-only loads (the kernel is
// bound by reading K once from HBM).  A unit's pages are split over CTAs of
// 256 pages, each of which forms the window mean itself (the window rows are
// read from L2 after the first); the page minima and maxima stay packed
// bf16 pairs until the dot product.
#include <cuda_runtime.h>

#include <cstdint>

#include "device_common.cuh"
#include "internal.h"

namespace rolekv {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kInFlight = 8;        // key-row loads a lane issues before using them
constexpr int kPagesPerCta = 256;   // pages of one unit handled by one CTA

__device__ __forceinline__ uint4 load_nc(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Elementwise min / max of two packed bf16 pairs (exact).
__device__ __forceinline__ uint32_t min_bf16x2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("min.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ uint32_t max_bf16x2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// The two bf16 halves of a 32-bit word, exactly, as fp32.
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__global__ void __launch_bounds__(kThreads, 3) quest_kernel(const QuestArgs a, int ctas_per_unit) {
  __shared__ float qpart[kThreads / 8][8 * 8 + 1];   // [row group][dims of a 16-byte chunk ...]
  __shared__ float qbar[128];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int u = blockIdx.x / ctas_per_unit;
  const int part = blockIdx.x % ctas_per_unit;
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
  const int npages = (n + a.page - 1) / a.page;
  const int p_begin = part * kPagesPerCta;
  if (p_begin >= npages) return;                   // (uniform)
  const int p_end = npages - p_begin < kPagesPerCta ? npages : p_begin + kPagesPerCta;
  const int d = a.d;
  const int CR = d / 8;                            // 16-byte chunks per row
#ifdef ROLEKV_CHECKED
  // Checked build: the unit's window queries, key rows and score row lie
  // inside the extents the call's shapes give, or the CTA returns (quest_score
  // has no status word to report it in).
  {
    const int w_eff = a.W < n ? a.W : n;
    const int64_t q0 = l * a.q_layer + s * a.q_seq + static_cast<int64_t>(h) * a.G * a.q_head;
    const int64_t k0 = l * a.k_layer + (a.varlen ? tok0 * a.k_tok : s * a.k_seq) + h * a.k_head;
    const int64_t s0 =
        a.varlen ? (static_cast<int64_t>(l) * a.Hkv + h) * a.T + tok0 : static_cast<int64_t>(u) * a.n_max;
    if (!(w_eff == 0 || in_bounds(q0, (a.G - 1) * a.q_head + (w_eff - 1) * a.q_tok + d, a.ext_q, nullptr)) ||
        !in_bounds(k0, (n - 1) * a.k_tok + d, a.ext_k, nullptr) || !in_bounds(s0, n, a.ext_scores, nullptr))
      return;                                      // (uniform)
  }
#endif

  // ---- mean of the window rows (the last W_eff positions of the G heads):
  // thread (row group rg, chunk c) sums chunk c of rows rg, rg + RG, ...
  {
    const int w_eff = a.W < n ? a.W : n;
    const int rows = a.G * w_eff;
    const int RG = kThreads / CR;
    const int c = tid % CR, rg = tid / CR;
    float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    for (int r = rg; r < rows; r += RG) {
      const int g = r / w_eff, i = r % w_eff;
      const int64_t o = l * a.q_layer + s * a.q_seq + static_cast<int64_t>(h * a.G + g) * a.q_head +
                        i * a.q_tok;
      const uint4 v = __ldg(reinterpret_cast<const uint4*>(a.q + o) + c);
      const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        acc[2 * j] += bf16_lo(w[j]);
        acc[2 * j + 1] += bf16_hi(w[j]);
      }
    }
    // qpart[rg][c*8 + j] holds row group rg's sum of dim c*8 + j (d <= 128:
    // CR * 8 = d values per row group, RG = 256 / CR groups)
    float* qp = &qpart[0][0];
    const int stride = 8 * 8 + 1;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int dim = c * 8 + j;
      // row group rg, dim -> flat slot; RG * d = 2048 floats at most
      const int flat = rg * d + dim;
      qp[(flat / 64) * stride + (flat % 64)] = acc[j];
    }
    __syncthreads();
    if (tid < d) {
      float t = 0.f;
      for (int g = 0; g < RG; ++g) {
        const int flat = g * d + tid;
        t += qp[(flat / 64) * stride + (flat % 64)];
      }
      qbar[tid] = t / static_cast<float>(rows);
    }
    __syncthreads();
  }

  // ---- page bounds: lane (tk, c) reads 16-byte chunk c of tokens tk, tk+TPI, ...
  const int TPI = 32 / CR;                         // tokens per warp-wide load
  const int c = lane % CR, tk = lane / CR;
  float qv[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) qv[j] = qbar[c * 8 + j];
  const uint16_t* kb = a.k + l * a.k_layer + (a.varlen ? tok0 * a.k_tok : s * a.k_seq) + h * a.k_head;
  const int64_t sbase =
      a.varlen ? (static_cast<int64_t>(l) * a.Hkv + h) * a.T + tok0 : static_cast<int64_t>(u) * a.n_max;
  for (int p = p_begin + warp; p < p_end; p += kWarps) {
    const int t0 = p * a.page;
    const int t1 = (n - t0 < a.page) ? n : t0 + a.page;
    // +inf / -inf as bf16 pairs
    uint32_t lo[4] = {0x7F807F80u, 0x7F807F80u, 0x7F807F80u, 0x7F807F80u};
    uint32_t hi[4] = {0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u};
    for (int t = t0 + tk; t < t1; t += TPI * kInFlight) {
      uint4 v[kInFlight];
#pragma unroll
      for (int x = 0; x < kInFlight; ++x) {
        const int tt = t + x * TPI;
        if (tt < t1) v[x] = load_nc(reinterpret_cast<const uint4*>(kb + tt * a.k_tok) + c);
      }
#pragma unroll
      for (int x = 0; x < kInFlight; ++x) {
        if (t + x * TPI < t1) {
          const uint32_t w[4] = {v[x].x, v[x].y, v[x].z, v[x].w};
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            lo[j] = min_bf16x2(lo[j], w[j]);
            hi[j] = max_bf16x2(hi[j], w[j]);
          }
        }
      }
    }
    // lanes holding the same chunk for other tokens
    for (int o = CR; o < 32; o <<= 1) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        lo[j] = min_bf16x2(lo[j], __shfl_xor_sync(0xffffffffu, lo[j], o));
        hi[j] = max_bf16x2(hi[j], __shfl_xor_sync(0xffffffffu, hi[j], o));
      }
    }
    float bound = 0.f;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      bound += fmaxf(qv[2 * j] * bf16_lo(lo[j]), qv[2 * j] * bf16_lo(hi[j]));
      bound += fmaxf(qv[2 * j + 1] * bf16_hi(lo[j]), qv[2 * j + 1] * bf16_hi(hi[j]));
    }
    for (int o = 1; o < CR; o <<= 1) bound += __shfl_xor_sync(0xffffffffu, bound, o);
    for (int x = t0 + lane; x < t1; x += 32) a.scores[sbase + x] = bound;
  }
}

}  // namespace

cudaError_t launch_quest(const QuestArgs& a, cudaStream_t stream) {
  if (a.n_units == 0 || a.n_max == 0) return cudaSuccess;
  const int max_pages = (a.n_max + a.page - 1) / a.page;
  const int ctas_per_unit = (max_pages + kPagesPerCta - 1) / kPagesPerCta;
  const int64_t grid = static_cast<int64_t>(a.n_units) * ctas_per_unit;
  quest_kernel<<<static_cast<unsigned>(grid), kThreads, 0, stream>>>(a, ctas_per_unit);
  return cudaGetLastError();
}

}  // namespace rolekv
