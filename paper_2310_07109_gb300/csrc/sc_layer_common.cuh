// sc_layer_common.cuh -- device helpers shared by the per-layer attention
// kernels (the paired rows kernel, the single-pass band kernel and the cols
// kernel): the resolved per-layer fields, TMA loads of 128-row tiles and of
// the global rows, the QK^T / PV tcgen05 issue sequences, bounded waits, warp
// reductions.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "sc_internal.cuh"
#include "sm103_primitives.cuh"

namespace sc {

// ---------------------------------------------------------------------------
// small helpers
// ---------------------------------------------------------------------------
// Barrier over the four warps of softmax warpgroup X (ids 2 and 3).
__device__ __forceinline__ void named_sync_wg(int X) {
  asm volatile("bar.sync %0, 128;" ::"r"(2 + X) : "memory");
}

__device__ __forceinline__ void named_sync_softmax() {
  asm volatile("bar.sync 1, 128;" ::: "memory");
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Bounded wait that ignores the abort flag: used in teardown to make sure no
// asynchronous copy or MMA is still writing into this CTA's memory.
__device__ __forceinline__ void drain_wait(uint64_t* bar, uint32_t parity) {
  int dummy = 0;
  mbar_wait(bar, parity, &dummy, 1000000000ull);
}

// Wait used by the softmax warps: the outcome is made uniform across the warp
// so that an expired wait can never leave lanes diverged at a warp vote.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort));
}

// The per-layer fields of this launch: as given, or (device-driven layer
// loop) the layer-0 values advanced to layer *dev_layer.
__device__ __forceinline__ LayerView layer_view(const LayerParams& p) {
  LayerView v;
  if (p.dev_layer == nullptr) {
    v.layer = p.layer; v.src_base = p.src_base;
    v.len = p.len; v.len_out = p.len_out; v.pos = p.pos; v.pos_out = p.pos_out;
    v.gcur = p.gcur; v.gcur_out = p.gcur_out; v.ng = p.ng; v.ng_out = p.ng_out;
    v.ident = p.ident; v.ident_out = p.ident_out;
    v.O = p.O; v.scores = p.scores; v.alpha = p.alpha;
    return v;
  }
  const int l = __ldcg(p.dev_layer);
  const bool odd = (l & 1) != 0;
  v.layer = l;
  v.src_base = l * p.tok_stride;
  v.len = p.len + static_cast<size_t>(l) * p.len_stride;
  v.len_out = p.len_out + static_cast<size_t>(l) * p.len_stride;
  v.pos = p.pos + l * p.row_stride;
  v.pos_out = p.pos_out + l * p.row_stride;
  v.gcur = odd ? p.gcur_out : p.gcur;
  v.gcur_out = odd ? const_cast<int32_t*>(p.gcur) : p.gcur_out;
  v.ng = odd ? p.ng_out : p.ng;
  v.ng_out = odd ? const_cast<int32_t*>(p.ng) : p.ng_out;
  v.ident = odd ? p.ident_out : p.ident;
  v.ident_out = odd ? const_cast<int32_t*>(p.ident) : p.ident_out;
  v.O = p.O != nullptr ? p.O + l * p.o_stride : (l == p.n_layers - 1 ? p.O_last : nullptr);
  v.scores = p.scores + l * p.row_stride;
  v.alpha = p.alphas[l];
  return v;
}

// Sequence b has been handed to the cluster kernel for this and later layers
// (its length here may be stale: read nothing else of it).
__device__ __forceinline__ bool owned_by_tail(const LayerParams& p, const LayerView& v, int b) {
  return p.tail_from != nullptr && __ldcg(p.tail_from + b) <= v.layer;
}

// Which source holds the current rows of sequence b, and the token index of
// its current row 0 in that source.
struct RowSource {
  int s;
  long long tok_b;
};

__device__ __forceinline__ RowSource row_source(const LayerParams& p, const LayerView& v, int b) {
  const bool id = __ldcg(v.ident + b) != 0;
  return {id ? 0 : 1, (id ? v.src_base : 0) + static_cast<long long>(b) * p.L};
}

// One 128-token tile (current rows c0 .. c0+127) of tensor t (0 Q, 1 K, 2 V)
// for head h: a single TMA copy.  Rows past the sequence are read but masked.
__device__ __forceinline__ void load_tile(const TensorMaps& m, int t, const RowSource& rs, int h,
                                          int c0, uint8_t* dst, uint64_t* bar) {
  tma_load_3d(dst, &m.tile[rs.s][t], 0, h, static_cast<int>(rs.tok_b + c0), bar);
}

// The 16 global rows (current indices gc[0..ng-1], the last repeated): lanes
// 0..3 gather four rows each.
__device__ __forceinline__ void load_globals(const TensorMaps& m, int t, const RowSource& rs, int h,
                                             int H, const int* gc, int ng, uint8_t* dst,
                                             uint64_t* bar, int lane) {
  if (lane < 4) {
    int r[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int g = min(4 * lane + k, ng - 1);
      r[k] = static_cast<int>((rs.tok_b + gc[g]) * H + h);
    }
    tma_gather4(dst + 512 * lane, &m.row[rs.s][t], 0, r[0], r[1], r[2], r[3], bar);
  }
}

// Issue D[128 x N] (+)= A[128 x 64] * B[N x 64]^T with both operands K-major
// 128B-swizzled tiles (A rows and B rows are 128-byte lines).
__device__ __forceinline__ void mma_qk(uint32_t d_tmem, uint32_t a_smem, uint32_t b_smem, int N) {
  const uint32_t idesc = (N == 128) ? idesc_bf16(128, 128, false, false)
                                    : idesc_bf16(128, 16, false, false);
#pragma unroll
  for (int k = 0; k < kHeadDim / 16; ++k)
    umma_bf16(d_tmem, sdesc_sw128(a_smem + 32 * k), sdesc_sw128(b_smem + 32 * k), idesc, k > 0);
}

// Issue D[128 x 64] (+)= P[128 x 16*ksteps] * V[16*ksteps x 64]: P is a K-major
// 128B-swizzled tile in two 64-key halves of 16 KB, V an MN-major tile of
// 128-byte key rows.
// P (A, K-major, 64-key blocks p_block bytes apart) from shared memory.
__device__ __forceinline__ void mma_pv(uint32_t d_tmem, uint32_t p_smem, uint32_t p_block,
                                       uint32_t v_smem, int ksteps, bool accumulate) {
  const uint32_t idesc = idesc_bf16(128, 64, false, true);
  for (int k = 0; k < ksteps; ++k)
    umma_bf16(d_tmem, sdesc_sw128(p_smem + (k >> 2) * p_block + (k & 3) * 32),
              sdesc_sw128(v_smem + k * 2048), idesc, (accumulate || k > 0) ? 1u : 0u);
}

// Issue P V for one 128-key tile: P (A) from tensor memory, V (B) MN-major smem.
__device__ __forceinline__ void mma_pv_ts(uint32_t d_tmem, uint32_t p_tmem, uint32_t v_smem,
                                          int ksteps, bool accumulate) {
  const uint32_t idesc = idesc_bf16(128, 64, false, true);
  for (int k = 0; k < ksteps; ++k)
    umma_bf16_ts(d_tmem, p_tmem + 8 * k, sdesc_sw128(v_smem + k * 2048), idesc,
                 (accumulate || k > 0) ? 1u : 0u);
}

// Bits lo..hi (inclusive, clipped to 0..31) of a 32-bit word; 0 when empty.
__device__ __forceinline__ uint32_t bit_range32(int lo, int hi) {
  lo = max(lo, 0);
  hi = min(hi, 31);
  return hi < lo ? 0u : ((0xffffffffu >> (31 - hi)) & (0xffffffffu << lo));
}

// Reduce 16 values per lane over the warp (butterfly reduce-scatter, 16
// shuffles): lane L returns the warp-wide result for element L >> 1.
template <typename Op>
__device__ __forceinline__ float warp_reduce16(float (&v)[16], Op op) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int half = 8, bit = 16; half >= 1; half >>= 1, bit >>= 1) {
    const bool upper = (lane & bit) != 0;
#pragma unroll
    for (int k = 0; k < half; ++k) {
      const float send = upper ? v[k] : v[k + half];
      const float keep = upper ? v[k + half] : v[k];
      v[k] = op(keep, __shfl_xor_sync(0xffffffffu, send, bit));
    }
  }
  return op(v[0], __shfl_xor_sync(0xffffffffu, v[0], 1));
}

struct OpAdd {
  __device__ __forceinline__ float operator()(float a, float b) const { return a + b; }
};
struct OpMax {
  __device__ __forceinline__ float operator()(float a, float b) const { return fmaxf(a, b); }
};

}  // namespace sc
