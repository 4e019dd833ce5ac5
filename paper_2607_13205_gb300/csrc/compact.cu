// Gather-compaction of the retained K/V rows into a dense cache (Section 6:
// the compacting implementation that realises the 1-B memory reduction).
// Each kept slot j of a unit copies row keep_idx[j] of K and of V; a row is
// d*2 bytes and is moved by d/8 lanes with 16-byte read-only loads and
// streaming stores, so a warp moves 32*16 = 512 contiguous-per-row bytes per
// instruction and every HBM sector it touches is used whole.
#include <cuda_runtime.h>

#include <cstdint>

#include "device_common.cuh"
#include "internal.h"

namespace rolekv {
namespace {

constexpr int kThreads = 256;
constexpr int kRowsPerBlock = 64;

__device__ __forceinline__ uint4 load_nc(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ void store_cs(uint4* p, uint4 v) {
  asm volatile("st.global.cs.v4.u32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y),
               "r"(v.z), "r"(v.w)
               : "memory");
}

__global__ void __launch_bounds__(kThreads) compact_kernel(const CompactArgs a, int chunks) {
  const int u = blockIdx.x / chunks;
  const int chunk = blockIdx.x % chunks;
  const int h = u % a.Hkv;
  const int s = (u / a.Hkv) % a.b;
  const int l = u / (a.Hkv * a.b);
  int n;
  int64_t tok0, kbase, K_s;
  if (a.varlen) {
    tok0 = a.cu_seqlens[s];
    n = a.cu_seqlens[s + 1] - a.cu_seqlens[s];
    // prefix of kept slots over the earlier sequences
    __shared__ int64_t cu_kept;
    if (threadIdx.x < 32) {
      int64_t part = 0;
      for (int x = threadIdx.x; x < s; x += 32)
        part += kept_rows(a.cu_seqlens[x + 1] - a.cu_seqlens[x], a.budget_fx, a.kept_extra);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
      if (threadIdx.x == 0) cu_kept = part;
    }
    __syncthreads();
    kbase = (static_cast<int64_t>(l) * a.Hkv + h) * a.Ktot + cu_kept;
    K_s = kept_rows(n, a.budget_fx, a.kept_extra);
  } else {
    tok0 = 0;
    n = a.n_max;
    kbase = static_cast<int64_t>(u) * a.K_dense;
    K_s = a.K_dense;
  }
  const int64_t kb = l * a.k_layer + (a.varlen ? tok0 * a.k_tok : s * a.k_seq) + h * a.k_head;
  const int64_t vb = l * a.v_layer + (a.varlen ? tok0 * a.v_tok : s * a.v_seq) + h * a.v_head;
  const int lanes_per_row = a.d / 8;              // 16-byte pieces per row
  const int rows_per_pass = kThreads / lanes_per_row;
  const int piece = threadIdx.x % lanes_per_row;
  const int j_begin = chunk * kRowsPerBlock;
  const int j_end = static_cast<int>(K_s < j_begin + kRowsPerBlock ? K_s : j_begin + kRowsPerBlock);
  for (int j = j_begin + threadIdx.x / lanes_per_row; j < j_end; j += rows_per_pass) {
    const int64_t slot = kbase + j;
    if (!in_bounds(slot, 1, a.ext_keep, a.status)) continue;
    const int32_t idx = a.keep_idx[slot];
    uint4 kv = make_uint4(0, 0, 0, 0), vv = make_uint4(0, 0, 0, 0);
    if (idx >= 0 && idx < n) {
      if (in_bounds(kb + idx * a.k_tok + piece * 8, 8, a.ext_k, a.status))
        kv = load_nc(reinterpret_cast<const uint4*>(a.k + kb + idx * a.k_tok) + piece);
      if (in_bounds(vb + idx * a.v_tok + piece * 8, 8, a.ext_v, a.status))
        vv = load_nc(reinterpret_cast<const uint4*>(a.v + vb + idx * a.v_tok) + piece);
    } else if (idx >= n && a.status != nullptr && piece == 0) {
      atomicOr(a.status, ROLEKV_STATUS_BAD_INDEX);
    }
    if (!in_bounds(slot, 1, a.ext_out_rows, a.status)) continue;
    store_cs(reinterpret_cast<uint4*>(a.k_out + slot * a.d) + piece, kv);
    store_cs(reinterpret_cast<uint4*>(a.v_out + slot * a.d) + piece, vv);
  }
}

}  // namespace

cudaError_t launch_compact(const CompactArgs& a, cudaStream_t stream) {
  if (a.n_units == 0 || a.K_max == 0) return cudaSuccess;
  const int chunks = (a.K_max + kRowsPerBlock - 1) / kRowsPerBlock;
  const int64_t grid = static_cast<int64_t>(a.n_units) * chunks;
  compact_kernel<<<static_cast<unsigned>(grid), kThreads, 0, stream>>>(a, chunks);
  return cudaGetLastError();
}

}  // namespace rolekv
