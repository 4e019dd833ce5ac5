// One decode step of attention through the compacted cache (Section 6: the
// 1-B memory and latency reduction that compaction exists for): for every
// (layer, sequence, KV head) and each of its G query heads,
//   o_g = sum_j softmax_j(scale q_g . k_j) v_j
// over the unit's cache rows (the kept slots; -1 slots of an infeasible budget
// are skipped; with budget 1 and no index the full cache).  Memory-bound: the
// cache rows are read once.  Split-K: CTA (unit, split) takes up to 1024 rows
// (a unit's splits equal in length).  A producer warp streams them into two
// shared-memory stages of 64 K rows and 64 V rows.  K goes through a tensor
// map, one copy per 64-column half of a stage, 128-byte swizzled so that the
// consumers' fragment loads stay conflict-free; V goes in one copy per stage
// (a bulk copy when the rows are contiguous, a tensor-map copy when they are
// strided, as in a packed varlen cache).  Layouts a tensor map cannot
// describe fall back to one bulk copy per row (K rows padded by 16 bytes).
// Each of four consumer warps takes 16 rows of a stage:
// the G x 16 dot products are one m16n8k16 bf16 MMA tile per 16 dimensions
// (cache rows x query heads padded to 8, fp32 accumulate), so no cross-lane
// reduction is needed; the online softmax (log2 units) runs in that fragment
// layout, and the probabilities and rescale factors pass through a per-warp
// shared buffer to the output accumulation, where the lanes run over the head
// dimension with packed f32x2 FMAs.  Every wait is a bounded mbarrier wait.
// The warps merge through shared memory; a second launch merges the splits of
// each (unit, head).
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "device_common.cuh"
#include "internal.h"

namespace rolekv {
namespace {

// DPL consecutive bf16 values: raw bits, then fp32.
template <int DPL>
struct RawDims {
  uint32_t w[DPL / 2];
};

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
    part += kept_rows(a.cu_seqlens[x + 1] - a.cu_seqlens[x], a.budget_fx, a.kept_extra);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
  return part;
}

constexpr int kDecWarps = 4;       // consumer warps per CTA
constexpr int kStages = 2;         // shared-memory stages of cache rows
constexpr int kTileRows = 16;      // rows of one MMA tile (one consumer warp)
constexpr int kStageRows = kDecWarps * kTileRows;
constexpr int kDecThreads = (kDecWarps + 1) * 32;   // + one producer warp

// K rows sit 16 bytes apart beyond their length, so that the eight rows read
// by one fragment load fall in different banks; V rows are packed.
__host__ __device__ constexpr int k_stride_bytes(int d) { return 2 * d + 16; }
__host__ __device__ constexpr int decode_smem_bytes(int d) {
  return kStages * kStageRows * (k_stride_bytes(d) + 2 * d);
}
// With K through a tensor map (KT): a stage's K rows in 64-column halves of
// kStageRows x 128 bytes each, 128-byte swizzled (the 16-byte chunk index of
// row r XOR-ed with r mod 8), which keeps the fragment loads conflict-free
// without padding; 1 KB of room to align the stages to the swizzle's 1 KB.
__host__ __device__ constexpr int decode_smem_bytes_kt(int d) {
  return kStages * kStageRows * (2 * d + 2 * d) + 1024;
}

__device__ __forceinline__ uint32_t lds32(const uint8_t* p) { return *reinterpret_cast<const uint32_t*>(p); }

// D = A B + D for one 16 x 8 x 16 bf16 tile (fp32 accumulate): A = 16 cache
// rows x 16 dims, B = 16 dims x 8 query heads.
__device__ __forceinline__ void mma16816(float* c, uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
      "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Consumer warps: q . k for 16 rows x 8 (padded) heads on the tensor cores,
// in the fragment layout (lane = 4 g + t holds rows g and g + 8 of heads 2t
// and 2t + 1); the online softmax runs there; the probabilities and rescale
// factors then go through a small per-warp shared buffer to the output
// accumulation, where the lanes run over the head dimension (DPL each).
template <int DPL, int GM, bool KT>
__global__ void __launch_bounds__(kDecThreads) decode_partial_kernel(const DecodeArgs a,
                                                                     const __grid_constant__ CUtensorMap k_map,
                                                                     const __grid_constant__ CUtensorMap v_map) {
  constexpr int D = DPL * 32;
  constexpr int KS = D / 16;                                // MMA k-steps
  constexpr int KSTR = KT ? 2 * D : k_stride_bytes(D);      // bytes of K per row in a stage
  constexpr int VSTR = 2 * D;
  constexpr int KHALF = kStageRows * 128;                   // KT: one 64-column half of a stage
  extern __shared__ __align__(128) uint8_t stage_raw[];     // K stages, then V stages
  uint8_t* stage_mem = KT ? stage_raw + ((1024u - (static_cast<uint32_t>(__cvta_generic_to_shared(stage_raw)) & 1023u)) & 1023u)
                          : stage_raw;
  __shared__ uint64_t full_bar[kStages], empty_bar[kStages];
  __shared__ int abort_flag;
  __shared__ float red[kDecWarps][GM][2];                   // per-warp (max2, sum) per head
  __shared__ __align__(16) float pbuf[kDecWarps][kTileRows][8];
  __shared__ __align__(16) float fbuf[kDecWarps][8];
  __shared__ float okbuf[kDecWarps][kTileRows];
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
  const int m = static_cast<int>(kept_rows(n, a.budget_fx, a.kept_extra));
  const int r0 = split * a.rows_per_split;
  if (r0 >= m) return;                              // (uniform: no partial is read)
  const int r1 = (m - r0 < a.rows_per_split) ? m : r0 + a.rows_per_split;
  const int nst = (r1 - r0 + kStageRows - 1) / kStageRows;
  const int64_t kb = l * a.k_layer + (a.varlen ? row0 * a.k_tok : s * a.k_seq) + h * a.k_head;
  const int64_t vb = l * a.v_layer + (a.varlen ? row0 * a.v_tok : s * a.v_seq) + h * a.v_head;
  uint8_t* ks = stage_mem;
  uint8_t* vs = stage_mem + kStages * kStageRows * KSTR;
#ifdef ROLEKV_CHECKED
  // Checked build: this split's K and V rows, kept indices, the group's
  // queries and its partials lie inside the extents the call's shapes give,
  // or the CTA returns before any copy is issued.
  {
    const int64_t i0 = a.varlen ? (static_cast<int64_t>(l) * a.Hkv + h) * a.Ktot + row0
                                : static_cast<int64_t>(u) * a.K_dense;
    const int64_t q0 = l * a.q_layer + s * a.q_seq + static_cast<int64_t>(h) * G * a.q_head;
    const int64_t p0 = (static_cast<int64_t>(u) * a.n_splits + split) * G * (a.d + 2);
    if (!(in_bounds(kb + r0 * a.k_tok, (r1 - r0 - 1) * a.k_tok + a.d, a.ext_k, nullptr) &&
          in_bounds(vb + r0 * a.v_tok, (r1 - r0 - 1) * a.v_tok + a.d, a.ext_v, nullptr) &&
          (a.keep_idx == nullptr || in_bounds(i0 + r0, r1 - r0, a.ext_keep, nullptr)) &&
          in_bounds(q0, (G - 1) * a.q_head + a.d, a.ext_q, nullptr) &&
          in_bounds(p0, static_cast<int64_t>(G) * (a.d + 2), a.ext_part, nullptr))) {
      if (threadIdx.x == 0 && a.status != nullptr) atomicOr(a.status, ROLEKV_STATUS_BOUNDS);
      return;
    }
  }
#endif

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], kDecWarps);
    }
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();

  // fragment-layout state: heads 2t, 2t+1 of this lane's rows
  const int g = lane >> 2, t = lane & 3;
  float mx[2] = {-INFINITY, -INFINITY}, sm[2] = {0.f, 0.f};
  // output accumulators: lanes over dims
  float2 acc[GM][DPL / 2];
#pragma unroll
  for (int hh = 0; hh < GM; ++hh)
#pragma unroll
    for (int i = 0; i < DPL / 2; ++i) acc[hh][i] = make_float2(0.f, 0.f);

  if (warp == kDecWarps) {
    // ---------------------------------------------------------- producer
    const bool vc = a.v_tok == D;                   // V rows contiguous
    int issued = 0;
    for (int st = 0; st < nst; ++st) {
      const int slot = st % kStages;
      bool ok = true;
      if (lane == 0) ok = mbar_wait(&empty_bar[slot], ((st / kStages) & 1) ^ 1, &abort_flag, a.status);
      if (!__shfl_sync(0xffffffffu, static_cast<int>(ok), 0)) break;
      const int rs = r0 + st * kStageRows;
      const int nr = (r1 - rs < kStageRows) ? r1 - rs : kStageRows;
      // (strided V rows: one tensor-map copy of the whole stage, kStageRows
      // rows whatever nr is -- the rows past the unit are not used)
      const uint32_t vbytes = static_cast<uint32_t>((a.v_tma ? kStageRows : nr) * VSTR);
      const uint32_t kbytes = static_cast<uint32_t>((KT ? kStageRows : nr) * VSTR);
      if (lane == 0) mbar_arrive_expect_tx(&full_bar[slot], kbytes + vbytes);
      __syncwarp();
      uint8_t* kd = ks + slot * kStageRows * KSTR;
      uint8_t* vd = vs + slot * kStageRows * VSTR;
      if constexpr (KT) {
        // the whole stage, one tensor-map copy per 64-column half (the rows
        // past the unit are not used)
        if (lane == 0) {
          const int64_t e0 = kb + static_cast<int64_t>(rs) * a.k_tok;
#pragma unroll
          for (int hf = 0; hf < D / 64; ++hf)
            tma_load_2d(kd + hf * KHALF, &k_map, static_cast<int32_t>(e0 % a.k_tok) + hf * 64,
                        static_cast<int32_t>(e0 / a.k_tok), &full_bar[slot]);
        }
      } else {
        for (int r = lane; r < nr; r += 32)
          bulk_copy_g2s(kd + r * KSTR, a.k + kb + static_cast<int64_t>(rs + r) * a.k_tok, VSTR, &full_bar[slot]);
      }
      if (a.v_tma) {
        if (lane == 0) {
          const int64_t e0 = vb + static_cast<int64_t>(rs) * a.v_tok;   // first element of the stage
          tma_load_2d(vd, &v_map, static_cast<int32_t>(e0 % a.v_tok), static_cast<int32_t>(e0 / a.v_tok),
                      &full_bar[slot]);
        }
      } else if (vc) {
        if (lane == 0) bulk_copy_g2s(vd, a.v + vb + static_cast<int64_t>(rs) * a.v_tok, nr * VSTR, &full_bar[slot]);
      } else {
        for (int r = lane; r < nr; r += 32)
          bulk_copy_g2s(vd + r * VSTR, a.v + vb + static_cast<int64_t>(rs + r) * a.v_tok, VSTR, &full_bar[slot]);
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
    // B fragments of the query heads (head g of the group, zero past G)
    uint32_t qb[KS][2];
    {
      const uint16_t* qp = a.q + l * a.q_layer + s * a.q_seq + static_cast<int64_t>(h * G + (g < G ? g : 0)) * a.q_head;
#pragma unroll
      for (int k = 0; k < KS; ++k) {
        qb[k][0] = g < G ? __ldg(reinterpret_cast<const uint32_t*>(qp + k * 16 + 2 * t)) : 0u;
        qb[k][1] = g < G ? __ldg(reinterpret_cast<const uint32_t*>(qp + k * 16 + 2 * t + 8)) : 0u;
      }
    }
    const int32_t* idx = nullptr;
    if (a.keep_idx != nullptr)
      idx = a.keep_idx + (a.varlen ? (static_cast<int64_t>(l) * a.Hkv + h) * a.Ktot + row0
                                   : static_cast<int64_t>(u) * a.K_dense);
    const float c1 = a.c1;
    const int d0 = lane * DPL;
    float* pw = &pbuf[warp][0][0];
    // kept-index words of this lane's two rows, loaded one stage ahead so that
    // their latency hides behind the stage before
    auto load_idx = [&](int stt, int32_t& ia, int32_t& ib) {
      const int trr = r0 + stt * kStageRows + warp * kTileRows;
      ia = (idx != nullptr && trr + g < r1) ? __ldg(idx + trr + g) : 0;
      ib = (idx != nullptr && trr + g + 8 < r1) ? __ldg(idx + trr + g + 8) : 0;
    };
    int32_t ia_cur, ib_cur;
    load_idx(0, ia_cur, ib_cur);
    for (int st = 0; st < nst; ++st) {
      const int slot = st % kStages;
      int32_t ia_next = 0, ib_next = 0;
      if (st + 1 < nst) load_idx(st + 1, ia_next, ib_next);
      const bool got = mbar_wait(&full_bar[slot], (st / kStages) & 1, &abort_flag, a.status);
      if (!__all_sync(0xffffffffu, got)) break;
      const int32_t ia = ia_cur, ib = ib_cur;
      ia_cur = ia_next;
      ib_cur = ib_next;
      const int tr0 = r0 + st * kStageRows + warp * kTileRows;   // first row of this warp's tile
      const uint8_t* kt = ks + slot * kStageRows * KSTR + warp * kTileRows * (KT ? 128 : KSTR);
      const uint8_t* vt = vs + slot * kStageRows * VSTR + warp * kTileRows * VSTR;
      if (tr0 < r1) {                                            // (uniform)
        float c[4] = {0.f, 0.f, 0.f, 0.f};
        if constexpr (KT) {
          // row g (and g + 8) of the warp's 16, swizzled: chunk c of a
          // 128-byte row sits at chunk c ^ (row mod 8) = c ^ g
          const uint8_t* kr = kt + g * 128 + 4 * t;
#pragma unroll
          for (int k = 0; k < KS; ++k) {
            const uint8_t* kh = kr + (k >> 2) * KHALF;
            const int c0 = 2 * (k & 3);
            const int o0 = ((c0 ^ g) << 4), o1 = (((c0 + 1) ^ g) << 4);
            mma16816(c, lds32(kh + o0), lds32(kh + 8 * 128 + o0), lds32(kh + o1), lds32(kh + 8 * 128 + o1),
                     qb[k][0], qb[k][1]);
          }
        } else {
          const uint8_t* ka = kt + g * KSTR + 4 * t;
#pragma unroll
          for (int k = 0; k < KS; ++k)
            mma16816(c, lds32(ka + 32 * k), lds32(ka + 8 * KSTR + 32 * k), lds32(ka + 32 * k + 16),
                     lds32(ka + 8 * KSTR + 32 * k + 16), qb[k][0], qb[k][1]);
        }
        // rows g and g + 8: inside the split, and a kept slot
        const int ra = tr0 + g, rb = tr0 + g + 8;
        const bool oka = ra < r1 && (idx == nullptr || ia >= 0);
        const bool okb = rb < r1 && (idx == nullptr || ib >= 0);
        const float s0 = oka ? c[0] * c1 : -INFINITY, s1 = oka ? c[1] * c1 : -INFINITY;
        const float s2 = okb ? c[2] * c1 : -INFINITY, s3 = okb ? c[3] * c1 : -INFINITY;
        float tm0 = fmaxf(s0, s2), tm1 = fmaxf(s1, s3);
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
          tm0 = fmaxf(tm0, __shfl_xor_sync(0xffffffffu, tm0, o));
          tm1 = fmaxf(tm1, __shfl_xor_sync(0xffffffffu, tm1, o));
        }
        const float mn0 = fmaxf(mx[0], tm0), mn1 = fmaxf(mx[1], tm1);
        const float f0 = mn0 == -INFINITY ? 1.f : fast_exp2(mx[0] - mn0);
        const float f1 = mn1 == -INFINITY ? 1.f : fast_exp2(mx[1] - mn1);
        const float p0 = mn0 == -INFINITY ? 0.f : fast_exp2(s0 - mn0);
        const float p1 = mn1 == -INFINITY ? 0.f : fast_exp2(s1 - mn1);
        const float p2 = mn0 == -INFINITY ? 0.f : fast_exp2(s2 - mn0);
        const float p3 = mn1 == -INFINITY ? 0.f : fast_exp2(s3 - mn1);
        sm[0] = sm[0] * f0 + (p0 + p2);
        sm[1] = sm[1] * f1 + (p1 + p3);
        mx[0] = mn0;
        mx[1] = mn1;
        *reinterpret_cast<float2*>(pw + g * 8 + 2 * t) = make_float2(p0, p1);
        *reinterpret_cast<float2*>(pw + (g + 8) * 8 + 2 * t) = make_float2(p2, p3);
        if (g == 0) *reinterpret_cast<float2*>(&fbuf[warp][2 * t]) = make_float2(f0, f1);
        if (t == 0) {
          okbuf[warp][g] = oka ? 1.f : 0.f;
          okbuf[warp][g + 8] = okb ? 1.f : 0.f;
        }
        __syncwarp();
        // o_h = o_h f_h + sum_j p_hj v_j, lanes over dims
        {
          const float4 F0 = *reinterpret_cast<const float4*>(&fbuf[warp][0]);
          float F[8] = {F0.x, F0.y, F0.z, F0.w, 1.f, 1.f, 1.f, 1.f};
          if (GM > 4) {
            const float4 F1 = *reinterpret_cast<const float4*>(&fbuf[warp][4]);
            F[4] = F1.x; F[5] = F1.y; F[6] = F1.z; F[7] = F1.w;
          }
#pragma unroll
          for (int hh = 0; hh < GM; ++hh)
#pragma unroll
            for (int i = 0; i < DPL / 2; ++i) acc[hh][i] = __fmul2_rn(acc[hh][i], make_float2(F[hh], F[hh]));
        }
        const bool all_ok = __all_sync(0xffffffffu, oka && okb);
#pragma unroll 4
        for (int j = 0; j < kTileRows; ++j) {
          float vr[DPL];
          unpack<DPL>(*reinterpret_cast<const RawDims<DPL>*>(vt + j * VSTR + d0 * 2), vr);
          // rows past the end hold stale shared memory: their values are
          // zeroed (a weight of zero would not remove a stale NaN)
          if (!all_ok) {
            const bool okj = okbuf[warp][j] != 0.f;
#pragma unroll
            for (int i = 0; i < DPL; ++i) vr[i] = okj ? vr[i] : 0.f;
          }
          const float4 P0 = *reinterpret_cast<const float4*>(pw + j * 8);
          float P[8] = {P0.x, P0.y, P0.z, P0.w, 0.f, 0.f, 0.f, 0.f};
          if (GM > 4) {
            const float4 P1 = *reinterpret_cast<const float4*>(pw + j * 8 + 4);
            P[4] = P1.x; P[5] = P1.y; P[6] = P1.z; P[7] = P1.w;
          }
#pragma unroll
          for (int hh = 0; hh < GM; ++hh)
#pragma unroll
            for (int i = 0; i < DPL / 2; ++i)
              acc[hh][i] = __ffma2_rn(make_float2(P[hh], P[hh]), make_float2(vr[2 * i], vr[2 * i + 1]), acc[hh][i]);
        }
        __syncwarp();                                              // pbuf is rewritten next tile
      }
      if (lane == 0) mbar_arrive(&empty_bar[slot]);
    }
    // per-head sums over the lanes of a head column (g = 0..7)
#pragma unroll
    for (int o = 4; o < 32; o <<= 1) {
      sm[0] += __shfl_xor_sync(0xffffffffu, sm[0], o);
      sm[1] += __shfl_xor_sync(0xffffffffu, sm[1], o);
    }
    if (g == 0) {
      if (2 * t < GM) {
        red[warp][2 * t][0] = mx[0];
        red[warp][2 * t][1] = sm[0];
      }
      if (2 * t + 1 < GM) {
        red[warp][2 * t + 1][0] = mx[1];
        red[warp][2 * t + 1][1] = sm[1];
      }
    }
  }
  __syncthreads();   // every stage consumed, every copy landed: the stages are free
  float* racc = reinterpret_cast<float*>(stage_mem);          // [warp][head][D]
  if (warp < kDecWarps) {
    const int d0 = lane * DPL;
#pragma unroll
    for (int hh = 0; hh < GM; ++hh)
#pragma unroll
      for (int i = 0; i < DPL / 2; ++i) {
        racc[(warp * GM + hh) * D + d0 + 2 * i] = acc[hh][i].x;
        racc[(warp * GM + hh) * D + d0 + 2 * i + 1] = acc[hh][i].y;
      }
  }
  __syncthreads();
  if (warp < kDecWarps) {
    const int d0 = lane * DPL;
    for (int gg = warp; gg < G; gg += kDecWarps) {
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < kDecWarps; ++w) M = fmaxf(M, red[w][gg][0]);
      float L = 0.f, o[DPL];
#pragma unroll
      for (int i = 0; i < DPL; ++i) o[i] = 0.f;
      if (M > -INFINITY) {
#pragma unroll
        for (int w = 0; w < kDecWarps; ++w) {
          const float mw = red[w][gg][0];
          if (mw == -INFINITY) continue;
          const float f = exp2f(mw - M);
          L += f * red[w][gg][1];
#pragma unroll
          for (int i = 0; i < DPL; ++i) o[i] += f * racc[(w * GM + gg) * D + d0 + i];
        }
      }
      float* out = a.part + ((static_cast<int64_t>(u) * a.n_splits + split) * a.G + gg) * (a.d + 2);
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
  const int m = static_cast<int>(kept_rows(n, a.budget_fx, a.kept_extra));
  const int ns = (m + a.rows_per_split - 1) / a.rows_per_split;
  const float* base = a.part + (static_cast<int64_t>(u) * a.n_splits * a.G + g) * (a.d + 2);
  const int64_t stride = static_cast<int64_t>(a.G) * (a.d + 2);
  const int64_t dst0 = l * a.o_layer + s * a.o_seq + static_cast<int64_t>(h * a.G + g) * a.o_head;
  if (!in_bounds(base - a.part, (ns > 0 ? (ns - 1) * stride : 0) + a.d + 2, a.ext_part, a.status) ||
      !in_bounds(dst0, a.d, a.ext_out, a.status))
    return;                                          // (checked build only)
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

template <int DPL, bool KT>
cudaError_t launch_decode_dk(const DecodeArgs& a, const CUtensorMap& kmap, const CUtensorMap& vmap,
                             cudaStream_t stream) {
  const int64_t grid1 = static_cast<int64_t>(a.n_units) * a.n_splits;
  const int64_t warps2 = static_cast<int64_t>(a.n_units) * a.G;
  const unsigned grid2 = static_cast<unsigned>((warps2 * 32 + 255) / 256);
  const int smem = KT ? decode_smem_bytes_kt(a.d) : decode_smem_bytes(a.d);
  cudaError_t e;
  if (grid1 == 0) {                                  // no rows anywhere: the merge writes zeros
    decode_combine_kernel<DPL><<<grid2, 256, 0, stream>>>(a);
    return cudaGetLastError();
  }
  if (a.G <= 4) {
    e = cudaFuncSetAttribute(decode_partial_kernel<DPL, 4, KT>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    decode_partial_kernel<DPL, 4, KT><<<static_cast<unsigned>(grid1), kDecThreads, smem, stream>>>(a, kmap, vmap);
  } else {
    e = cudaFuncSetAttribute(decode_partial_kernel<DPL, 8, KT>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    decode_partial_kernel<DPL, 8, KT><<<static_cast<unsigned>(grid1), kDecThreads, smem, stream>>>(a, kmap, vmap);
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  decode_combine_kernel<DPL><<<grid2, 256, 0, stream>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_decode(const DecodeArgs& a, const CUtensorMap& kmap, const CUtensorMap& vmap,
                          cudaStream_t stream) {
  if (a.n_units == 0) return cudaSuccess;
  if (a.k_tma)
    return a.d == 128 ? launch_decode_dk<4, true>(a, kmap, vmap, stream)
                      : launch_decode_dk<2, true>(a, kmap, vmap, stream);
  return a.d == 128 ? launch_decode_dk<4, false>(a, kmap, vmap, stream)
                    : launch_decode_dk<2, false>(a, kmap, vmap, stream);
}

}  // namespace rolekv
