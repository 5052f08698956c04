// sc_encoder.cu -- device code of the encoder layer around the sparse
// attention: the projections and the feed-forward block as tcgen05 GEMMs with
// a row gather on the A operand, and the post-layer norms.
//
// RoBERTa-style post-LN layer (the encoder SparseCoder prunes, Fig.
// "sparsecoder"), hidden size D = 64 H, on the n current tokens of a sequence:
//   Q, K, V = X W_{q,k,v}^T + b                     (one GEMM, N = 3D, split output)
//   O, s, keep = sparse attention + token pruning   (sc_kernels.cu)
//   S1 = X[kept] + O[kept] W_o^T + b_o              (GEMM: A and the residual gathered
//                                                    by the kept tokens' current index)
//   H1 = LN(S1);  F = GELU(H1 W_1^T + b_1);  S2 = H1 + F W_2^T + b_2;  Y = LN(S2)
// so everything after the attention runs on the kept tokens only, and the
// compaction of the kept rows is the A-operand gather of the output
// projection (Y is the next layer's X, already compacted).
//
// GEMM: one CTA per 128 x 128 output tile of one sequence (rows are (sequence,
// row) pairs, row < rows[b] read on the device), K in steps of 64 through a
// three-stage TMA ring: A's 128 rows by four-row gathers (tile::gather4, any
// row order), W's 128 rows by one tiled copy, both 128B-swizzled and K-major;
// one thread issues the MMAs into a 128-column fp32 accumulator in tensor
// memory; four warps read it back and apply bias, GELU and the residual.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "sc_internal.cuh"
#include "sm103_primitives.cuh"

namespace sc {

constexpr int kGemmThreads = 192;   // warp 0 loads, warp 1 issues, warps 2-5 write back
constexpr int kGemmStages = 3;
constexpr int kGemmBK = 64;         // K per stage: one 128-byte swizzle atom of bf16
constexpr uint32_t kGemmStageBytes = 2 * kTileBytes;   // A and W tiles, 16 KB each
constexpr uint32_t kGemmDyn = kGemmStages * kGemmStageBytes + 1024;

struct GemmSmem {
  uint64_t full[kGemmStages], empty[kGemmStages], done;
  uint32_t tmem_base;
  int abort;
  float bias[kTile];
};

// Bounded wait that ignores the abort flag (teardown: no copy or MMA may still
// write into this CTA's memory when it exits).
__device__ __forceinline__ void drain_wait_gemm(uint64_t* bar, uint32_t parity) {
  int dummy = 0;
  mbar_wait(bar, parity, &dummy, 1000000000ull);
}

__device__ __forceinline__ bool warp_wait_gemm(uint64_t* bar, uint32_t parity, volatile int* abort) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort));
}

__device__ __forceinline__ uint16_t bf16_bits(float x) {
  return __bfloat16_as_ushort(__float2bfloat16_rn(x));
}

__device__ __forceinline__ float gelu_erf(float x) {
  return 0.5f * x * (1.f + erff(x * 0.70710678118654752f));
}

__global__ void __launch_bounds__(kGemmThreads, 2)
    sc_gemm_kernel(const __grid_constant__ GemmParams p) {
  pdl_wait();
  pdl_launch_dependents();
  const int n0 = blockIdx.x * kTile;
  const int tiles_per_seq = (p.L + kTile - 1) / kTile;
  const int b = blockIdx.y / tiles_per_seq, r0 = (blockIdx.y % tiles_per_seq) * kTile;
  const int rows = p.rows ? min(__ldcg(p.rows + b), p.L) : p.L;
  if (r0 >= rows) return;

  extern __shared__ uint8_t dyn_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dyn_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ GemmSmem sm;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int ksteps = p.K / kGemmBK;

  if (tid == 0) {
    for (int s = 0; s < kGemmStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    mbar_init(&sm.done, 1);
    sm.abort = 0;
    fence_mbar_init();
  }
  if (tid < kTile) sm.bias[tid] = p.bias ? __ldg(p.bias + n0 + tid) : 0.f;
  if (warp == 1) tmem_alloc(&sm.tmem_base, 128);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = sm.tmem_base;
  volatile int* abort_flag = &sm.abort;

  if (warp == 0) {
    // ------------------------------------------------------------- loads
    // this lane's four A rows (rows past the sequence read row 0: discarded)
    int ar[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int r = r0 + 4 * lane + k;
      const int src = r < rows ? (p.gidx ? __ldcg(p.gidx + static_cast<size_t>(b) * p.L + r) : r) : 0;
      ar[k] = b * p.L + src;
    }
    bool ok = true;
    for (int kt = 0, s = 0, use = 0; ok && kt < ksteps; ++kt) {
      if (kt >= kGemmStages) ok = warp_wait_gemm(&sm.empty[s], (use - 1) & 1, abort_flag);
      if (!ok) break;
      uint8_t* As = base + s * kGemmStageBytes;
      uint8_t* Ws = As + kTileBytes;
      if (lane == 0) {
        mbar_arrive_expect_tx(&sm.full[s], kGemmStageBytes);
        tma_load_2d(Ws, &p.map_w, kt * kGemmBK, n0, &sm.full[s]);
      }
      __syncwarp();
      tma_gather4(As + 512 * lane, &p.map_a, kt * kGemmBK, ar[0], ar[1], ar[2], ar[3], &sm.full[s]);
      if (++s == kGemmStages) {
        s = 0;
        ++use;
      }
    }
    // nothing may still be landing in shared memory when the CTA exits
    if (lane == 0)
      for (int s = 0; s < kGemmStages && s < ksteps; ++s) {
        const int last = s + kGemmStages * ((ksteps - 1 - s) / kGemmStages);
        drain_wait_gemm(&sm.full[s], (last / kGemmStages) & 1);
      }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------- MMA issue
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(128, 128, false, false);
      bool ok = true;
      for (int kt = 0, s = 0, use = 0; ok && kt < ksteps; ++kt) {
        if (!(ok = mbar_wait(&sm.full[s], use & 1, abort_flag))) break;
        tc_fence_after();
        const uint32_t a = smem_u32(base + s * kGemmStageBytes), w = a + kTileBytes;
#pragma unroll
        for (int k = 0; k < kGemmBK / 16; ++k)
          umma_bf16(tm, sdesc_sw128(a + 32 * k), sdesc_sw128(w + 32 * k), idesc, (kt | k) != 0);
        umma_commit(&sm.empty[s]);   // the stage is free once these MMAs are done
        if (++s == kGemmStages) {
          s = 0;
          ++use;
        }
      }
      umma_commit(&sm.done);
      drain_wait_gemm(&sm.done, 0);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------- write back
    const int q = warp & 3;                   // tensor-memory lane quarter of this warp
    const int r = r0 + 32 * q + lane;         // output row of this thread
    const bool valid = r < rows;
    const bool ok = warp_wait_gemm(&sm.done, 0, abort_flag);
    const size_t orow = static_cast<size_t>(b) * p.L + r;
    const int rsrc = valid ? (p.res_gathered && p.gidx ? __ldcg(p.gidx + static_cast<size_t>(b) * p.L + r) : r) : 0;
    const uint16_t* res = p.res ? p.res + (static_cast<size_t>(b) * p.L + rsrc) * p.N + n0 : nullptr;
    // output block of this tile (split outputs: column blocks of out_split)
    int nb = n0, ldo = p.N;
    void* outp = p.out;
    if (p.out_split > 0) {
      const int j = n0 / p.out_split;
      outp = p.outs[j];
      nb = n0 - j * p.out_split;
      ldo = p.out_split;
    }
    if (ok) tc_fence_after();
#pragma unroll 1
    for (int c = 0; c < kTile; c += 32) {
      float v[32];
      tmem_ld32(tm + (static_cast<uint32_t>(32 * q) << 16) + c, v);
      tmem_ld_wait();
      if (!ok || !valid) continue;
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        float x = v[k] + sm.bias[c + k];
        if (p.gelu) x = gelu_erf(x);
        v[k] = x;
      }
      if (res) {
#pragma unroll
        for (int k = 0; k < 32; k += 8) {
          const uint4 u = __ldcg(reinterpret_cast<const uint4*>(res + c + k));
          const uint32_t w4[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            v[k + 2 * e] += __uint_as_float(w4[e] << 16);
            v[k + 2 * e + 1] += __uint_as_float(w4[e] & 0xffff0000u);
          }
        }
      }
      if (p.out_f32) {
        float* o = static_cast<float*>(outp) + orow * ldo + nb + c;
#pragma unroll
        for (int k = 0; k < 32; k += 4)
          *reinterpret_cast<float4*>(o + k) = make_float4(v[k], v[k + 1], v[k + 2], v[k + 3]);
      } else {
        uint16_t* o = static_cast<uint16_t*>(outp) + orow * ldo + nb + c;
#pragma unroll
        for (int k = 0; k < 32; k += 8)
          *reinterpret_cast<uint4*>(o + k) =
              make_uint4(pack_bf16x2(v[k], v[k + 1]), pack_bf16x2(v[k + 2], v[k + 3]),
                         pack_bf16x2(v[k + 4], v[k + 5]), pack_bf16x2(v[k + 6], v[k + 7]));
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tm, 128);
  }
  if (tid == 0 && sm.abort) atomicOr(p.status, kStatusTimeout);
}

// ---------------------------------------------------------------------------
// layer norm over D features, one warp per row: fp32 in, bf16 out
// ---------------------------------------------------------------------------
constexpr int kLnThreads = 256;
constexpr int kLnMaxPer = 32;   // features per lane: D <= 1024

__global__ void __launch_bounds__(kLnThreads)
    sc_layernorm_kernel(const __grid_constant__ LayerNormParams p) {
  pdl_wait();
  pdl_launch_dependents();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long row = static_cast<long long>(blockIdx.x) * (kLnThreads / 32) + warp;
  if (row >= static_cast<long long>(p.B) * p.L) return;
  const int b = static_cast<int>(row / p.L), r = static_cast<int>(row % p.L);
  if (r >= (p.rows ? min(__ldcg(p.rows + b), p.L) : p.L)) return;
  const float* x = p.in + row * p.D;
  const int per = p.D / 32;   // features of this lane: lane, lane + 32, ...
  float v[kLnMaxPer];
  float s = 0.f;
#pragma unroll
  for (int k = 0; k < kLnMaxPer; ++k) {
    v[k] = k < per ? __ldcg(x + lane + 32 * k) : 0.f;
    s += v[k];
  }
  for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
  const float mean = s / static_cast<float>(p.D);
  float q = 0.f;
#pragma unroll
  for (int k = 0; k < kLnMaxPer; ++k)
    if (k < per) {
      const float d = v[k] - mean;
      q += d * d;
    }
  for (int off = 16; off > 0; off >>= 1) q += __shfl_xor_sync(0xffffffffu, q, off);
  const float inv = 1.f / sqrtf(q / static_cast<float>(p.D) + p.eps);
  uint16_t* y = p.out + row * p.D;
#pragma unroll
  for (int k = 0; k < kLnMaxPer; ++k)
    if (k < per) {
      const int f = lane + 32 * k;
      const float o = (v[k] - mean) * inv * __ldg(p.gamma + f) + __ldg(p.beta + f);
      y[f] = bf16_bits(o);
    }
}

// ---------------------------------------------------------------------------
// launch helpers used by the C ABI
// ---------------------------------------------------------------------------
cudaError_t configure_encoder() {
  return cudaFuncSetAttribute(sc_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(kGemmDyn));
}

template <typename... KArgs>
static cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t st, const KArgs&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

cudaError_t launch_gemm(const GemmParams& p, cudaStream_t st) {
  const int tiles_per_seq = (p.L + kTile - 1) / kTile;
  return launch_pdl(sc_gemm_kernel, dim3(p.N / kTile, p.B * tiles_per_seq), dim3(kGemmThreads),
                    kGemmDyn, st, p);
}

cudaError_t launch_layernorm(const LayerNormParams& p, cudaStream_t st) {
  const long long rows = static_cast<long long>(p.B) * p.L;
  const unsigned blocks = static_cast<unsigned>((rows + kLnThreads / 32 - 1) / (kLnThreads / 32));
  return launch_pdl(sc_layernorm_kernel, dim3(blocks), dim3(kLnThreads), 0, st, p);
}

}  // namespace sc
