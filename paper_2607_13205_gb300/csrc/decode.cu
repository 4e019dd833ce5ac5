// One decode step of attention through the compacted cache (Section 6: the
// 1-B memory and latency reduction that compaction exists for): for every
// (layer, sequence, KV head) and each of its G query heads,
//   o_g = sum_j softmax_j(scale q_g . k_j) v_j
// over the unit's cache rows (the kept slots; -1 slots of an infeasible budget
// are skipped; with budget 1 and no index the full cache).  Memory-bound: the
// cache rows are read once.  Split-K: CTA (unit, split) takes 512 rows.  A
// producer warp streams them into four shared-memory stages of 32 K rows and
// 32 V rows with bulk copies (one per stage when a unit's rows are
// contiguous, one per row otherwise), so the bytes in flight do not depend on
// registers; each of four consumer warps takes 8 rows of every stage for all
// G query heads, lanes over the head dimension: the G x rows dot products are
// reduced across the warp and an online softmax per head keeps (max, sum,
// unnormalised output) in log2 units.  Every wait is a bounded mbarrier wait.
// The warps merge through shared memory; a second launch merges the splits of
// each (unit, head).
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "device_common.cuh"
#include "internal.h"

namespace rolekv {
namespace {

constexpr int kRowBatch = 8;

__device__ __forceinline__ float bf16f(uint16_t x) { return __uint_as_float(static_cast<uint32_t>(x) << 16); }

// DPL consecutive bf16 values: raw bits, then fp32.
template <int DPL>
struct RawDims {
  uint32_t w[DPL / 2];
};

template <int DPL>
__device__ __forceinline__ RawDims<DPL> load_raw(const uint16_t* p) {
  RawDims<DPL> r;
  if constexpr (DPL == 4) {
    const uint2 v = __ldg(reinterpret_cast<const uint2*>(p));
    r.w[0] = v.x;
    r.w[1] = v.y;
  } else {
    r.w[0] = __ldg(reinterpret_cast<const uint32_t*>(p));
  }
  return r;
}

template <int DPL>
__device__ __forceinline__ void unpack(const RawDims<DPL>& r, float* out) {
#pragma unroll
  for (int i = 0; i < DPL / 2; ++i) {
    out[2 * i] = __uint_as_float(r.w[i] << 16);
    out[2 * i + 1] = __uint_as_float(r.w[i] & 0xFFFF0000u);
  }
}

__device__ __forceinline__ int64_t kept_prefix(const DecodeArgs& a, int s) {
  // kept rows of the sequences before s (varlen), by one warp
  int64_t part = 0;
  for (int x = threadIdx.x & 31; x < s; x += 32)
    part += kept_slots(a.cu_seqlens[x + 1] - a.cu_seqlens[x], a.budget_fx);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
  return part;
}

constexpr int kDecWarps = 4;       // consumer warps per CTA
constexpr int kStages = 4;         // shared-memory stages of cache rows
constexpr int kStageRows = 32;     // rows per stage (8 per consumer warp)
constexpr int kDecThreads = (kDecWarps + 1) * 32;   // + one producer warp

__host__ __device__ constexpr int decode_smem_bytes(int d) { return 2 * kStages * kStageRows * d * 2; }

template <int DPL, int GM>
__global__ void __launch_bounds__(kDecThreads) decode_partial_kernel(const DecodeArgs a) {
  constexpr int RB = GM <= 4 ? kRowBatch : kRowBatch / 2;   // rows per batch (registers)
  extern __shared__ __align__(128) uint8_t stage_mem[];     // K stages, then V stages
  __shared__ uint64_t full_bar[kStages], empty_bar[kStages];
  __shared__ int abort_flag;
  __shared__ float red[kDecWarps][GM][2];                   // per-warp (max2, sum) per head
  __shared__ float racc[kDecWarps][GM][128];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int u = blockIdx.x / a.n_splits;
  const int split = blockIdx.x % a.n_splits;
  const int h = u % a.Hkv;
  const int s = (u / a.Hkv) % a.b;
  const int l = u / (a.Hkv * a.b);
  const int G = a.G;
  int n;
  int64_t row0;                                     // first cache row of the unit (packed layouts)
  if (a.varlen) {
    n = a.cu_seqlens[s + 1] - a.cu_seqlens[s];
    row0 = kept_prefix(a, s);
  } else {
    n = a.n_max;
    row0 = 0;
  }
  const int m = static_cast<int>(kept_slots(n, a.budget_fx));
  const int r0 = split * a.rows_per_split;
  if (r0 >= m) return;                              // (uniform: no partial is read)
  const int r1 = (m - r0 < a.rows_per_split) ? m : r0 + a.rows_per_split;
  const int nst = (r1 - r0 + kStageRows - 1) / kStageRows;
  const int rowbytes = a.d * 2;
  const int64_t kb = l * a.k_layer + (a.varlen ? row0 * a.k_tok : s * a.k_seq) + h * a.k_head;
  const int64_t vb = l * a.v_layer + (a.varlen ? row0 * a.v_tok : s * a.v_seq) + h * a.v_head;
  uint8_t* ks = stage_mem;
  uint8_t* vs = stage_mem + kStages * kStageRows * rowbytes;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], kDecWarps);
    }
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();

  float mx[GM], sum[GM], acc[GM][DPL];
#pragma unroll
  for (int g = 0; g < GM; ++g) {
    mx[g] = -INFINITY;
    sum[g] = 0.f;
#pragma unroll
    for (int i = 0; i < DPL; ++i) acc[g][i] = 0.f;
  }

  if (warp == kDecWarps) {
    // ---------------------------------------------------------- producer
    const bool kc = a.k_tok == a.d, vc = a.v_tok == a.d;   // rows contiguous
    int issued = 0;
    for (int st = 0; st < nst; ++st) {
      const int slot = st % kStages;
      bool ok = true;
      if (lane == 0) ok = mbar_wait(&empty_bar[slot], ((st / kStages) & 1) ^ 1, &abort_flag, a.status);
      if (!__shfl_sync(0xffffffffu, static_cast<int>(ok), 0)) break;
      const int rs = r0 + st * kStageRows;
      const int nr = (r1 - rs < kStageRows) ? r1 - rs : kStageRows;
      if (lane == 0) mbar_arrive_expect_tx(&full_bar[slot], static_cast<uint32_t>(2 * nr * rowbytes));
      __syncwarp();
      uint8_t* kd = ks + slot * kStageRows * rowbytes;
      uint8_t* vd = vs + slot * kStageRows * rowbytes;
      if (kc) {
        if (lane == 0) bulk_copy_g2s(kd, a.k + kb + static_cast<int64_t>(rs) * a.k_tok, nr * rowbytes, &full_bar[slot]);
      } else if (lane < nr) {
        bulk_copy_g2s(kd + lane * rowbytes, a.k + kb + static_cast<int64_t>(rs + lane) * a.k_tok, rowbytes, &full_bar[slot]);
      }
      if (vc) {
        if (lane == 0) bulk_copy_g2s(vd, a.v + vb + static_cast<int64_t>(rs) * a.v_tok, nr * rowbytes, &full_bar[slot]);
      } else if (lane < nr) {
        bulk_copy_g2s(vd + lane * rowbytes, a.v + vb + static_cast<int64_t>(rs + lane) * a.v_tok, rowbytes, &full_bar[slot]);
      }
      ++issued;
    }
    // the copies still in flight land before the CTA leaves (bounded)
    if (lane == 0) {
      const int first = issued > kStages ? issued - kStages : 0;
      for (int st = first; st < issued; ++st)
        mbar_wait(&full_bar[st % kStages], (st / kStages) & 1, nullptr, nullptr);
    }
    __syncwarp();
  } else {
    // --------------------------------------------------------- consumers
    const int d0 = lane * DPL;
    float q[GM][DPL];
#pragma unroll
    for (int g = 0; g < GM; ++g) {
      const uint16_t* qp = a.q + l * a.q_layer + s * a.q_seq +
                           static_cast<int64_t>(h * G + (g < G ? g : 0)) * a.q_head + d0;
#pragma unroll
      for (int i = 0; i < DPL; ++i) q[g][i] = g < G ? bf16f(qp[i]) * a.c1 : 0.f;
    }
    const int32_t* idx = nullptr;
    if (a.keep_idx != nullptr)
      idx = a.keep_idx + (a.varlen ? (static_cast<int64_t>(l) * a.Hkv + h) * a.Ktot + row0
                                   : static_cast<int64_t>(u) * a.K_dense);
    for (int st = 0; st < nst; ++st) {
      const int slot = st % kStages;
      const bool got = mbar_wait(&full_bar[slot], (st / kStages) & 1, &abort_flag, a.status);
      if (!__all_sync(0xffffffffu, got)) break;
      const int rs = r0 + st * kStageRows;
      const uint8_t* kst = ks + slot * kStageRows * rowbytes + d0 * 2;
      const uint8_t* vst = vs + slot * kStageRows * rowbytes + d0 * 2;
#pragma unroll
      for (int half = 0; half < kStageRows / kDecWarps / RB; ++half) {
        const int jr0 = warp * (kStageRows / kDecWarps) + half * RB;   // row within the stage
        RawDims<DPL> kraw[RB], vraw[RB];
        bool ok[RB];
#pragma unroll
        for (int j = 0; j < RB; ++j) {
          const int r = rs + jr0 + j;
          ok[j] = r < r1 && (idx == nullptr || __ldg(idx + (r < r1 ? r : r1 - 1)) >= 0);
          kraw[j] = *reinterpret_cast<const RawDims<DPL>*>(kst + (jr0 + j) * rowbytes);
          vraw[j] = *reinterpret_cast<const RawDims<DPL>*>(vst + (jr0 + j) * rowbytes);
        }
        float sc[GM][RB];
#pragma unroll
        for (int j = 0; j < RB; ++j) {
          float kr[DPL];
          unpack<DPL>(kraw[j], kr);
#pragma unroll
          for (int g = 0; g < GM; ++g) {
            float t = 0.f;
#pragma unroll
            for (int i = 0; i < DPL; ++i) t = fmaf(q[g][i], kr[i], t);
            sc[g][j] = t;
          }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1)
#pragma unroll
          for (int g = 0; g < GM; ++g)
            if (g < G) {
#pragma unroll
              for (int j = 0; j < RB; ++j) sc[g][j] += __shfl_xor_sync(0xffffffffu, sc[g][j], o);
            }
        // rows past the end hold stale shared memory: their values are
        // zeroed (a weight of zero would not remove a stale NaN)
        float vr[RB][DPL];
#pragma unroll
        for (int j = 0; j < RB; ++j) {
          unpack<DPL>(vraw[j], vr[j]);
#pragma unroll
          for (int i = 0; i < DPL; ++i) vr[j][i] = ok[j] ? vr[j][i] : 0.f;
        }
#pragma unroll
        for (int g = 0; g < GM; ++g) {
          if (g >= G) continue;
          float bm = -INFINITY;
#pragma unroll
          for (int j = 0; j < RB; ++j) {
            if (!ok[j]) sc[g][j] = -INFINITY;
            bm = fmaxf(bm, sc[g][j]);
          }
          if (bm == -INFINITY) continue;            // (uniform) nothing valid here
          const float mn = fmaxf(mx[g], bm);
          const float rescale = fast_exp2(mx[g] - mn);
          sum[g] *= rescale;
#pragma unroll
          for (int i = 0; i < DPL; ++i) acc[g][i] *= rescale;
#pragma unroll
          for (int j = 0; j < RB; ++j) {
            const float p = ok[j] ? fast_exp2(sc[g][j] - mn) : 0.f;
            sum[g] += p;
#pragma unroll
            for (int i = 0; i < DPL; ++i) acc[g][i] = fmaf(p, vr[j][i], acc[g][i]);
          }
          mx[g] = mn;
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty_bar[slot]);
    }
    // this warp's state per head, for the merge
#pragma unroll
    for (int g = 0; g < GM; ++g) {
      if (lane == 0) {
        red[warp][g][0] = mx[g];
        red[warp][g][1] = sum[g];
      }
#pragma unroll
      for (int i = 0; i < DPL; ++i) racc[warp][g][d0 + i] = acc[g][i];
    }
  }
  __syncthreads();
  if (warp < kDecWarps) {
    const int d0 = lane * DPL;
    for (int g = warp; g < G; g += kDecWarps) {
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < kDecWarps; ++w) M = fmaxf(M, red[w][g][0]);
      float L = 0.f, o[DPL];
#pragma unroll
      for (int i = 0; i < DPL; ++i) o[i] = 0.f;
      if (M > -INFINITY) {
#pragma unroll
        for (int w = 0; w < kDecWarps; ++w) {
          const float mw = red[w][g][0];
          if (mw == -INFINITY) continue;
          const float f = exp2f(mw - M);
          L += f * red[w][g][1];
#pragma unroll
          for (int i = 0; i < DPL; ++i) o[i] += f * racc[w][g][d0 + i];
        }
      }
      float* out = a.part + ((static_cast<int64_t>(u) * a.n_splits + split) * a.G + g) * (a.d + 2);
#pragma unroll
      for (int i = 0; i < DPL; ++i) out[d0 + i] = o[i];
      if (lane == 0) {
        out[a.d] = M;
        out[a.d + 1] = L;
      }
    }
  }
}

// Merge of the splits of each (unit, query head): one warp, lanes over dims.
template <int DPL>
__global__ void __launch_bounds__(256) decode_combine_kernel(const DecodeArgs a) {
  const int64_t wid = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (wid >= static_cast<int64_t>(a.n_units) * a.G) return;
  const int u = static_cast<int>(wid / a.G), g = static_cast<int>(wid % a.G);
  const int h = u % a.Hkv;
  const int s = (u / a.Hkv) % a.b;
  const int l = u / (a.Hkv * a.b);
  const int n = a.varlen ? a.cu_seqlens[s + 1] - a.cu_seqlens[s] : a.n_max;
  const int m = static_cast<int>(kept_slots(n, a.budget_fx));
  const int ns = (m + a.rows_per_split - 1) / a.rows_per_split;
  const float* base = a.part + (static_cast<int64_t>(u) * a.n_splits * a.G + g) * (a.d + 2);
  const int64_t stride = static_cast<int64_t>(a.G) * (a.d + 2);
  float M = -INFINITY;
  for (int x = 0; x < ns; ++x) M = fmaxf(M, base[x * stride + a.d]);
  float L = 0.f, o[DPL];
#pragma unroll
  for (int i = 0; i < DPL; ++i) o[i] = 0.f;
  if (M > -INFINITY) {
    for (int x = 0; x < ns; ++x) {
      const float* p = base + x * stride;
      const float mxs = p[a.d];
      if (mxs == -INFINITY) continue;
      const float w = exp2f(mxs - M);
      L += w * p[a.d + 1];
#pragma unroll
      for (int i = 0; i < DPL; ++i) o[i] += w * p[lane * DPL + i];
    }
  }
  float* dst = a.out + l * a.o_layer + s * a.o_seq + static_cast<int64_t>(h * a.G + g) * a.o_head + lane * DPL;
#pragma unroll
  for (int i = 0; i < DPL; ++i) dst[i] = L > 0.f ? o[i] / L : 0.f;
}

// Diagnostic: the bounded mbarrier wait of the kernels above, on a phase that
// nothing completes, so that it runs out after limit_ns and records
// ROLEKV_STATUS_TIMEOUT; the CTA then returns normally.
__global__ void selftest_wait_kernel(uint64_t limit_ns, int32_t* status) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  mbar_wait_for(&bar, 0, nullptr, status, limit_ns);   // phase 0 never completes
}

}  // namespace

cudaError_t launch_selftest_wait(uint64_t limit_ns, int32_t* status, cudaStream_t stream) {
  selftest_wait_kernel<<<1, 32, 0, stream>>>(limit_ns, status);
  return cudaGetLastError();
}

template <int DPL>
cudaError_t launch_decode_d(const DecodeArgs& a, cudaStream_t stream) {
  const int64_t grid1 = static_cast<int64_t>(a.n_units) * a.n_splits;
  const int64_t warps2 = static_cast<int64_t>(a.n_units) * a.G;
  const unsigned grid2 = static_cast<unsigned>((warps2 * 32 + 255) / 256);
  const int smem = decode_smem_bytes(a.d);
  cudaError_t e;
  if (a.G <= 4) {
    e = cudaFuncSetAttribute(decode_partial_kernel<DPL, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    decode_partial_kernel<DPL, 4><<<static_cast<unsigned>(grid1), kDecThreads, smem, stream>>>(a);
  } else {
    e = cudaFuncSetAttribute(decode_partial_kernel<DPL, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    decode_partial_kernel<DPL, 8><<<static_cast<unsigned>(grid1), kDecThreads, smem, stream>>>(a);
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  decode_combine_kernel<DPL><<<grid2, 256, 0, stream>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t stream) {
  if (a.n_units == 0) return cudaSuccess;
  return a.d == 128 ? launch_decode_d<4>(a, stream) : launch_decode_d<2>(a, stream);
}

}  // namespace rolekv
