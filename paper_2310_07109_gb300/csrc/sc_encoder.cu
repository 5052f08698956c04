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
// GEMM: output tiles of 128 rows of one sequence (rows are (sequence, row)
// pairs, row < rows[b] read on the device) by 256, 192 or 128 columns (chosen
// on the host), one persistent CTA per SM walking the tiles; K in steps of 64
// through a four-stage TMA ring: A's 128 rows by one tiled copy, or by
// four-row gathers (tile::gather4, any row order) when A is gathered, W's rows
// by one tiled copy, both 128B-swizzled and K-major; one thread issues the
// MMAs (M = 128) into one of two 256-column fp32 accumulators in tensor memory
// while eight warps read the other back, apply bias, GELU and the residual,
// and store each 32-column chunk through shared memory as whole row segments.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cstdint>
#include <type_traits>

#include "sc_internal.cuh"
#include "sm103_primitives.cuh"

namespace sc {

constexpr int kGemmThreads = 320;   // warp 0 loads, warp 1 issues, warps 2-9 write back
constexpr int kGemmEpiWarps = 8;    // two per tensor-memory lane quarter, one column half each
constexpr int kGemmStages = 4;
constexpr int kGemmBK = 64;         // K per stage: one 128-byte swizzle atom of bf16
constexpr int kGemmBN = 256;        // most output columns per tile (one MMA, N <= 256)
constexpr uint32_t kGemmABytes = kTileBytes;              // 128 rows x 64
constexpr uint32_t kGemmWBytes = kGemmBN * kGemmBK * 2;   // 256 rows x 64
constexpr uint32_t kGemmStageBytes = kGemmABytes + kGemmWBytes;
// after the ring: a 4 KB staging area per write-back warp (32 rows of 128 bytes),
// through which the stores of a chunk leave as whole row segments
constexpr uint32_t kGemmStageOut = 4096;
constexpr uint32_t kGemmDyn = kGemmStages * kGemmStageBytes + kGemmEpiWarps * kGemmStageOut + 1024;

struct GemmSmem {
  uint64_t full[kGemmStages], empty[kGemmStages];
  uint64_t tfull[2], tempty[2];   // accumulator buffers: written by the MMAs, read back
  uint32_t tmem_base;
  int abort;
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

// GELU(x) = x/2 (1 + erf(x / sqrt 2)) with erf from Abramowitz & Stegun
// 7.1.26 (|error| <= 1.5e-7): erf(z) = 1 - (a1 t + ... + a5 t^5) exp(-z^2),
// t = 1 / (1 + p z), z >= 0, extended as an odd function.  With
// h = (1 - erf(|x| / sqrt 2)) / 2:  GELU(x) = x (1 - h) for x >= 0, x h below.
// Two values at once: the polynomial, the products and the exponent in packed
// fp32 pairs (the coefficients carry the factor 1/2), with
// exp(-z^2) = 2^(-z^2 log2 e).
__device__ __forceinline__ void gelu_erf2(float& x0, float& x1) {
  const float z0 = fabsf(x0) * 0.70710678118654752f, z1 = fabsf(x1) * 0.70710678118654752f;
  const uint64_t z = f2_pack(z0, z1);
  float d0, d1;
  f2_unpack(f2_fma(z, f2_pack(0.3275911f, 0.3275911f), f2_pack(1.f, 1.f)), d0, d1);
  const uint64_t t = f2_pack(__fdividef(1.f, d0), __fdividef(1.f, d1));
  uint64_t poly = f2_fma(f2_pack(0.5307027145f, 0.5307027145f), t,
                         f2_pack(-0.7265760135f, -0.7265760135f));
  poly = f2_fma(poly, t, f2_pack(0.7107068705f, 0.7107068705f));
  poly = f2_fma(poly, t, f2_pack(-0.142248368f, -0.142248368f));
  poly = f2_fma(poly, t, f2_pack(0.127414796f, 0.127414796f));
  float e0, e1;
  f2_unpack(f2_mul(f2_mul(z, z), f2_pack(-1.44269504088896341f, -1.44269504088896341f)), e0, e1);
  float h0, h1;
  f2_unpack(f2_mul(f2_mul(poly, t), f2_pack(ex2(e0), ex2(e1))), h0, h1);
  x0 *= x0 >= 0.f ? 1.f - h0 : h0;
  x1 *= x1 >= 0.f ? 1.f - h1 : h1;
}

// Tile t of the launch: column block nt of width bn (fastest, so that the
// CTAs of a wave share A rows), row tile rt of sequence b.
struct GemmTile {
  int b, r0, n0, nw, rows;
  bool skip;
};

__device__ __forceinline__ GemmTile gemm_tile(const GemmParams& p, int t) {
  const int tiles_n = (p.N + p.bn - 1) / p.bn;
  const int tiles_r = (p.L + kTile - 1) / kTile;
  GemmTile g;
  const int nt = t % tiles_n, rest = t / tiles_n;
  g.b = rest / tiles_r;
  g.r0 = (rest % tiles_r) * kTile;
  g.n0 = nt * p.bn;
  g.nw = min(p.bn, p.N - g.n0);
  g.rows = p.rows ? min(__ldcg(p.rows + g.b), p.L) : p.L;
  g.skip = g.r0 >= g.rows;
  return g;
}

// Persistent: each CTA walks tiles blockIdx.x, blockIdx.x + gridDim.x, ...;
// the accumulator alternates between two 256-column buffers, so that the
// write-back of one tile overlaps the MMAs of the next.
__global__ void __launch_bounds__(kGemmThreads, 1)
    sc_gemm_kernel(const __grid_constant__ GemmParams p) {
  pdl_wait();
  pdl_launch_dependents();
  extern __shared__ uint8_t dyn_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dyn_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ GemmSmem sm;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int ksteps = p.K / kGemmBK;
  const int tiles = p.B * ((p.L + kTile - 1) / kTile) * ((p.N + p.bn - 1) / p.bn);

  if (tid == 0) {
    for (int s = 0; s < kGemmStages; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&sm.tfull[a], 1);
      mbar_init(&sm.tempty[a], kGemmEpiWarps);   // one arrival per write-back warp
    }
    sm.abort = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(&sm.tmem_base, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = sm.tmem_base;
  volatile int* abort_flag = &sm.abort;

  if (warp == 0) {
    // ------------------------------------------------------------- loads
    bool ok = true;
    int s = 0, use = 0;
    for (int t = blockIdx.x; ok && t < tiles; t += gridDim.x) {
      const GemmTile g = gemm_tile(p, t);
      if (g.skip) continue;
      // gathered A: this lane's four rows (rows past the sequence read row 0:
      // discarded); otherwise one tiled copy of 128 consecutive rows
      int ar[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int r = g.r0 + 4 * lane + k;
        const int src =
            r < g.rows ? (p.a_idx ? __ldcg(p.a_idx + static_cast<size_t>(g.b) * p.L + r) : r) : 0;
        ar[k] = g.b * p.L + src;
      }
      const bool gather = p.a_idx != nullptr;
      for (int kt = 0; ok && kt < ksteps; ++kt) {
        if (use > 0 && !(ok = warp_wait_gemm(&sm.empty[s], (use - 1) & 1, abort_flag))) break;
        uint8_t* As = base + s * kGemmStageBytes;
        uint8_t* Ws = As + kGemmABytes;
        if (lane == 0) {
          mbar_arrive_expect_tx(&sm.full[s], kGemmABytes + p.wbox * kGemmBK * 2);
          tma_load_2d(Ws, &p.map_w, kt * kGemmBK, g.n0, &sm.full[s]);
          if (!gather) tma_load_2d(As, &p.map_at, kt * kGemmBK, g.b * p.L + g.r0, &sm.full[s]);
        }
        __syncwarp();
        if (gather)
          tma_gather4(As + 512 * lane, &p.map_a, kt * kGemmBK, ar[0], ar[1], ar[2], ar[3],
                      &sm.full[s]);
        if (++s == kGemmStages) {
          s = 0;
          ++use;
        }
      }
    }
    // nothing may still be landing in shared memory when the CTA exits: the
    // last fill of every slot
    if (lane == 0)
      for (int q = 0; q < kGemmStages; ++q) {
        const int fills = use + (q < s ? 1 : 0);
        if (fills > 0) drain_wait_gemm(&sm.full[q], (fills - 1) & 1);
      }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------------- MMA issue
    if (lane == 0) {
      bool ok = true;
      int s = 0, use = 0, j = 0;
      for (int t = blockIdx.x; ok && t < tiles; t += gridDim.x) {
        const GemmTile g = gemm_tile(p, t);
        if (g.skip) continue;
        const int acc = j & 1;
        // the buffer's previous tile has been read back
        if (j >= 2 && !(ok = mbar_wait(&sm.tempty[acc], ((j >> 1) - 1) & 1, abort_flag))) break;
        tc_fence_after();
        const uint32_t idesc = idesc_bf16(128, g.nw, false, false);
        const uint32_t d = tm + acc * kGemmBN;
        for (int kt = 0; ok && kt < ksteps; ++kt) {
          if (!(ok = mbar_wait(&sm.full[s], use & 1, abort_flag))) break;
          tc_fence_after();
          const uint32_t a = smem_u32(base + s * kGemmStageBytes), w = a + kGemmABytes;
#pragma unroll
          for (int k = 0; k < kGemmBK / 16; ++k)
            umma_bf16(d, sdesc_sw128(a + 32 * k), sdesc_sw128(w + 32 * k), idesc, (kt | k) != 0);
          umma_commit(&sm.empty[s]);   // the stage is free once these MMAs are done
          if (++s == kGemmStages) {
            s = 0;
            ++use;
          }
        }
        umma_commit(&sm.tfull[acc]);
        ++j;
      }
      // every MMA has completed before the tensor memory is freed
      uint64_t* last = &sm.empty[(s + kGemmStages - 1) % kGemmStages];
      if (use > 0 || s > 0) {
        const int q = (s + kGemmStages - 1) % kGemmStages;
        const int fills = use + (q < s ? 1 : 0);
        drain_wait_gemm(last, (fills - 1) & 1);
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------- write back
    const int q = warp & 3;                  // tensor-memory lane quarter of this warp
    const int ch = (warp - 2) / 4;           // column half of the tile
    uint8_t* const stg = base + kGemmStages * kGemmStageBytes + (warp - 2) * kGemmStageOut;
    bool ok = true;
    int j = 0;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x) {
      const GemmTile g = gemm_tile(p, t);
      if (g.skip) continue;
      const int acc = j & 1;
      const int r = g.r0 + 32 * q + lane;
      const bool in_rows = r < g.rows;
      const int rsrc =
          in_rows ? (p.res_idx ? __ldcg(p.res_idx + static_cast<size_t>(g.b) * p.L + r) : r) : 0;
      const uint16_t* res =
          p.res ? p.res + (static_cast<size_t>(g.b) * p.L + rsrc) * p.N + g.n0 : nullptr;
      const int cbeg = ch * (p.bn / 2), cend = min(g.nw, (ch + 1) * (p.bn / 2));
      // without GELU, this row's residual over the warp's first two chunks of
      // 32 columns is loaded before the accumulator is ready, so that its
      // latency overlaps the MMAs (later chunks, and GEMMs with GELU, load
      // theirs chunk by chunk)
      const bool res_ahead = res != nullptr && !p.gelu;
      uint4 rpf[2][4];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int c = cbeg + 32 * u;
#pragma unroll
        for (int k = 0; k < 4; ++k)
          rpf[u][k] = (res_ahead && c < cend)
                          ? __ldcg(reinterpret_cast<const uint4*>(res + c + 8 * k))
                          : make_uint4(0u, 0u, 0u, 0u);
      }
      ok = ok && warp_wait_gemm(&sm.tfull[acc], (j >> 1) & 1, abort_flag);
      const uint32_t rows_mask = __ballot_sync(0xffffffffu, ok && in_rows);
      const size_t orow0 = static_cast<size_t>(g.b) * p.L + g.r0 + 32 * q;   // the warp's row 0
      int nb = g.n0, ldo = p.N;
      void* outp = p.out;
      if (p.out_split > 0) {
        const int sj = g.n0 / p.out_split;
        outp = p.outs[sj];
        nb = g.n0 - sj * p.out_split;
        ldo = p.out_split;
      }
      tc_fence_after();
      // one 32-column chunk: bias, GELU (only where may_gelu is true), the
      // residual (rv: its 32 values, or nullptr: loaded here), store
      auto chunk = [&](int c, const uint4* rv, auto may_gelu) {
        float v[32];
        tmem_ld32(tm + acc * kGemmBN + (static_cast<uint32_t>(32 * q) << 16) + c, v);
        tmem_ld_wait();
        if (rows_mask == 0u) return;   // warp-uniform
        const float4* bp = reinterpret_cast<const float4*>(p.bias + g.n0 + c);
#pragma unroll
        for (int k = 0; k < 32; k += 4) {
          const float4 b4 = p.bias ? __ldg(bp + k / 4) : make_float4(0.f, 0.f, 0.f, 0.f);
          v[k] += b4.x;
          v[k + 1] += b4.y;
          v[k + 2] += b4.z;
          v[k + 3] += b4.w;
        }
        if constexpr (decltype(may_gelu)::value) {
          if (p.gelu)
#pragma unroll
            for (int k = 0; k < 32; k += 2) gelu_erf2(v[k], v[k + 1]);
        }
        if (res != nullptr) {
#pragma unroll
          for (int k = 0; k < 32; k += 8) {
            const uint4 r4 = rv != nullptr ? rv[k / 8]
                                           : __ldcg(reinterpret_cast<const uint4*>(res + c + k));
            const uint32_t w4[4] = {r4.x, r4.y, r4.z, r4.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              v[k + 2 * e] += __uint_as_float(w4[e] << 16);
              v[k + 2 * e + 1] += __uint_as_float(w4[e] & 0xffff0000u);
            }
          }
        }
        // the warp's 32 rows leave as whole 128-byte (fp32) or 64-byte (bf16)
        // row segments; rows past the sequence are not written
        if (p.out_f32) {
#pragma unroll
          for (int k = 0; k < 32; k += 4)
            stage_row_piece<8>(stg, k / 4,
                               make_uint4(__float_as_uint(v[k]), __float_as_uint(v[k + 1]),
                                          __float_as_uint(v[k + 2]), __float_as_uint(v[k + 3])));
          flush_staged_rows<8>(
              stg, reinterpret_cast<uint16_t*>(static_cast<float*>(outp) + orow0 * ldo + nb + c),
              2 * static_cast<size_t>(ldo), rows_mask);
        } else {
#pragma unroll
          for (int k = 0; k < 32; k += 8)
            stage_row_piece<4>(stg, k / 8,
                               make_uint4(pack_bf16x2(v[k], v[k + 1]), pack_bf16x2(v[k + 2], v[k + 3]),
                                          pack_bf16x2(v[k + 4], v[k + 5]),
                                          pack_bf16x2(v[k + 6], v[k + 7])));
          flush_staged_rows<4>(stg, static_cast<uint16_t*>(outp) + orow0 * ldo + nb + c,
                               static_cast<size_t>(ldo), rows_mask);
        }
      };
      if (!res_ahead) {
#pragma unroll 1
        for (int c = cbeg; c < cend; c += 32) chunk(c, nullptr, std::true_type{});
      } else {
        // unrolled, so that the prefetched residual stays in registers
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (cbeg + 32 * u < cend) chunk(cbeg + 32 * u, u < 2 ? rpf[u] : nullptr, std::false_type{});
      }
      // the buffer may take the tile after next
      tc_fence_before();
      warp_arrive(&sm.tempty[acc]);
      ++j;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tm, 512);
  }
  if (tid == 0 && sm.abort) atomicOr(p.status, kStatusTimeout);
}

// ---------------------------------------------------------------------------
// row gather: the kept rows of a bf16 matrix, consecutive (8 rows per CTA,
// 16-byte vectors, every load of a thread issued before its stores)
// ---------------------------------------------------------------------------
constexpr int kRgRows = 8;
constexpr int kRgThreads = 256;

__global__ void __launch_bounds__(kRgThreads)
    sc_row_gather_kernel(const __grid_constant__ RowGatherParams p) {
  pdl_launch_dependents();
  pdl_wait();
  const int b = blockIdx.y, r0 = blockIdx.x * kRgRows;
  const int n = __ldcg(p.rows + b);
  if (r0 >= n) return;
  const int cnt = min(kRgRows, n - r0);
  const int vec = p.D / 8;
  const int total = cnt * vec;
  constexpr int kPer = 4;
  const size_t base = static_cast<size_t>(b) * p.L;
  for (int k0 = threadIdx.x; k0 < total; k0 += kRgThreads * kPer) {
    uint4 v[kPer];
    size_t dofs[kPer];
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int k = k0 + u * kRgThreads;
      if (k < total) {
        const int rr = k / vec, e = k - rr * vec;
        const int src = __ldcg(p.idx + base + r0 + rr);
        v[u] = __ldcg(reinterpret_cast<const uint4*>(p.src + (base + src) * p.D) + e);
        dofs[u] = (base + r0 + rr) * vec + e;
      }
    }
#pragma unroll
    for (int u = 0; u < kPer; ++u)
      if (k0 + u * kRgThreads < total) reinterpret_cast<uint4*>(p.dst)[dofs[u]] = v[u];
  }
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
  uint16_t* y = p.out + row * p.D;
  if (p.vec) {
    // lane covers features 4 lane + 128 k .. + 3: 16-byte loads, 8-byte stores
    constexpr int kMaxChunks = kLnMaxPer / 4;
    const int chunks = p.D / 128;
    float4 v[kMaxChunks];
    float s = 0.f;
#pragma unroll
    for (int k = 0; k < kMaxChunks; ++k) {
      v[k] = k < chunks ? __ldcg(reinterpret_cast<const float4*>(x) + lane + 32 * k)
                        : make_float4(0.f, 0.f, 0.f, 0.f);
      s += (v[k].x + v[k].y) + (v[k].z + v[k].w);
    }
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    const float mean = s / static_cast<float>(p.D);
    float q = 0.f;
#pragma unroll
    for (int k = 0; k < kMaxChunks; ++k)
      if (k < chunks) {
        const float a = v[k].x - mean, b2 = v[k].y - mean, c = v[k].z - mean, d = v[k].w - mean;
        q += (a * a + b2 * b2) + (c * c + d * d);
      }
    for (int off = 16; off > 0; off >>= 1) q += __shfl_xor_sync(0xffffffffu, q, off);
    const float inv = 1.f / sqrtf(q / static_cast<float>(p.D) + p.eps);
#pragma unroll
    for (int k = 0; k < kMaxChunks; ++k)
      if (k < chunks) {
        const int f4 = lane + 32 * k;
        const float4 g = __ldg(reinterpret_cast<const float4*>(p.gamma) + f4);
        const float4 be = __ldg(reinterpret_cast<const float4*>(p.beta) + f4);
        const uint2 o = make_uint2(pack_bf16x2((v[k].x - mean) * inv * g.x + be.x,
                                               (v[k].y - mean) * inv * g.y + be.y),
                                   pack_bf16x2((v[k].z - mean) * inv * g.z + be.z,
                                               (v[k].w - mean) * inv * g.w + be.w));
        reinterpret_cast<uint2*>(y)[f4] = o;
      }
    return;
  }
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
  static int sms = 0;
  if (sms == 0) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
  }
  const long long tiles = static_cast<long long>(p.B) * ((p.L + kTile - 1) / kTile) *
                          ((p.N + p.bn - 1) / p.bn);
  const unsigned grid = static_cast<unsigned>(tiles < sms ? tiles : sms);
  return launch_pdl(sc_gemm_kernel, dim3(grid), dim3(kGemmThreads), kGemmDyn, st, p);
}

cudaError_t launch_row_gather(const RowGatherParams& p, cudaStream_t st) {
  dim3 grid((p.L + kRgRows - 1) / kRgRows, p.B);
  return launch_pdl(sc_row_gather_kernel, grid, dim3(kRgThreads), 0, st, p);
}

cudaError_t launch_layernorm(const LayerNormParams& p, cudaStream_t st) {
  const long long rows = static_cast<long long>(p.B) * p.L;
  const unsigned blocks = static_cast<unsigned>((rows + kLnThreads / 32 - 1) / (kLnThreads / 32));
  auto al = [](const void* q, unsigned a) { return (reinterpret_cast<uintptr_t>(q) % a) == 0; };
  LayerNormParams q = p;
  q.vec = (p.D % 128 == 0 && al(p.in, 16) && al(p.gamma, 16) && al(p.beta, 16) && al(p.out, 8))
              ? 1 : 0;
  return launch_pdl(sc_layernorm_kernel, dim3(blocks), dim3(kLnThreads), 0, st, q);
}

}  // namespace sc
