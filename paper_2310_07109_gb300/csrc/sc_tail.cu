// sc_tail.cu -- the remaining layers of a sequence once at most 256 tokens
// survive: one thread-block cluster per sequence, one CTA per head, every
// remaining layer in one launch.
//
// After the first layers have pruned a sequence, a layer is a few hundred
// tokens: far too little work to fill the GPU, so its time is the critical path
// of its kernels.  Here a layer of one head is a chain inside one CTA:
//
//   gather   Q, K, V rows of the current tokens (by original position; all
//            threads, 16-byte asynchronous copies) into 128B-swizzled tiles;
//            the rows of the next layer's candidates (a superset of its
//            tokens) are prefetched into L2
//   rows     S = Q K^T for the whole row (N <= 256 keys in tensor memory), an
//            exact two-pass softmax in fp32 (base 2), P (bf16) back to tensor
//            memory, O = P V, LSE_i
//   columns  S^T = K Q^T, and per key column j the sum over rows of
//            exp2(S_ij - LSE_i): one thread per column, no cross-thread sums
//   heads    the H CTAs exchange their column sums through distributed shared
//            memory; every CTA adds the heads in the same fixed order, so all
//            take the same keep decisions (s_j >= alpha_l / n, j == 0 kept) and
//            compact the token list the same way, without a second exchange
//
// The allowed set (window, global tokens), the softmax, the vertical
// accumulation and the order-preserving removal are those of Sec. "Sparse
// Attention", Sec. "Extractor of Attention Scores in Sparse Attention Matrix"
// and Sec. "Token Pruning"; global rows are ordinary rows here (all of their
// <= 256 keys are in tensor memory at once).
#include <cuda_runtime.h>
#include <cstdint>

#include "sc_internal.cuh"
#include "sm103_primitives.cuh"

namespace sc {

constexpr int kTailThreads = 288;                        // 2 softmax warpgroups + control warp
constexpr uint32_t kTailOpBytes = kTailMax * kHeadDim * 2;   // 256 rows of one tensor (32 KB)
// Q, K, V operands plus alignment; the remainder keeps a second CTA off the SM,
// since each CTA holds all 512 tensor-memory columns while it waits at cluster
// barriers (two CTAs of different clusters sharing an SM could otherwise wait
// on each other's allocation).
constexpr uint32_t kTailDyn = 120 * 1024;
static_assert(3 * kTailOpBytes + 1024 <= kTailDyn, "tail operands exceed the dynamic shared memory");

struct TailSmem {
  uint64_t bar_free[2], bar_fin;
  uint64_t bar_s[2], bar_p[2], bar_o[2], bar_st[2];
  uint32_t tmem_base;
  int abort;
  int n[2];
  int wcnt[8];
  int gpos[kMaxGlobal];               // global positions (sorted), -1 past n_global
  uint32_t gbits[2][kTailMax / 32];   // global flags of the current / next token list
  int32_t pos[2][kTailMax];           // original positions of the current / next tokens
  alignas(16) float nlse[kTailMax];   // -LSE of each query row (-inf past n)
  float colsum[2][kTailMax];          // this head's column sums, by layer parity
};

__device__ __forceinline__ bool tail_is_global(const TailSmem& sm, int ps) {
  bool g = false;
#pragma unroll
  for (int k = 0; k < kMaxGlobal; ++k) g |= (sm.gpos[k] == ps);
  return g;
}

__device__ __forceinline__ void tail_named_sync() {
  asm volatile("bar.sync 1, 256;" ::: "memory");
}

__device__ __forceinline__ bool tail_wait(uint64_t* bar, uint32_t parity, volatile int* abort) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort));
}

// Bits a..b (inclusive, clipped to 0..31) of a 32-bit word.
__device__ __forceinline__ uint32_t bit_range(int a, int b) {
  a = max(a, 0);
  b = min(b, 31);
  return b < a ? 0u : ((0xffffffffu >> (31 - b)) & (0xffffffffu << a));
}

// Allowed partners of one token (query row, or key column) among the 32
// tokens of chunk q: inside its window [lo, hi] (already clipped to the
// sequence), global partners, everything when the token itself is global;
// never past the sequence end.  The relation is symmetric, so the same mask
// serves the row softmax and the column sums.
struct Partners {
  int lo, hi;       // window, current indices
  bool all;         // token is global, or the window covers the sequence
  bool valid;       // token < n
};

__device__ __forceinline__ uint32_t partner_mask(const Partners& t, const TailSmem& sm, int cur,
                                                 int q, int n) {
  const int c0 = 32 * q;
  const uint32_t inseq = bit_range(0, n - 1 - c0);
  if (!t.valid) return 0u;
  if (t.all) return inseq;
  return (bit_range(t.lo - c0, t.hi - c0) | sm.gbits[cur][q]) & inseq;
}

// x[k] = -inf where bit k of m is clear; skipped when the whole warp's masks are full
__device__ __forceinline__ void apply_mask(float* x, uint32_t m) {
  if (__all_sync(0xffffffffu, m == 0xffffffffu)) return;
#pragma unroll
  for (int k = 0; k < 32; ++k) x[k] = ((m >> k) & 1u) ? x[k] : -INFINITY;
}

__global__ void __launch_bounds__(kTailThreads, 1)
    sc_tail_kernel(const __grid_constant__ TailParams p) {
  const int H = p.H, w = p.w, L = p.L, B = p.B, n_layers = p.n_layers;
  const int h = static_cast<int>(blockIdx.x) % H, b = static_cast<int>(blockIdx.x) / H;
  // every CTA of the cluster reads the same values: the exits below are uniform
  const int l0 = __ldcg(p.tail_from + b);
  if (l0 >= n_layers) return;
  const int n0 = __ldcg(p.len + static_cast<size_t>(l0) * B + b);
  if (n0 <= 0 || n0 > kTailMax) {
    if (h == 0 && threadIdx.x == 0) {
      if (n0 > kTailMax) atomicOr(p.status, kStatusInternal);
      else
        for (int l = l0; l < n_layers; ++l) p.len[static_cast<size_t>(l + 1) * B + b] = 0;
    }
    return;
  }

  extern __shared__ uint8_t dyn_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dyn_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ TailSmem sm;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // rows that are not loaded in a layer still enter MMAs whose results are
  // masked or discarded: they must hold finite values
  for (int k = tid; k < static_cast<int>(3 * kTailOpBytes / 16); k += kTailThreads)
    reinterpret_cast<uint4*>(base)[k] = make_uint4(0u, 0u, 0u, 0u);
  if (tid == 0) {
    mbar_init(&sm.bar_free[0], 128);
    mbar_init(&sm.bar_free[1], 128);
    mbar_init(&sm.bar_fin, 1);
    for (int X = 0; X < 2; ++X) {
      mbar_init(&sm.bar_s[X], 1);
      mbar_init(&sm.bar_p[X], 128);
      mbar_init(&sm.bar_o[X], 1);
      mbar_init(&sm.bar_st[X], 1);
    }
    sm.abort = 0;
    sm.n[0] = n0;
    fence_mbar_init();
  }
  if (tid < kMaxGlobal) sm.gpos[tid] = tid < p.n_global ? p.global_pos[tid] : -1;
  if (warp == 8) tmem_alloc(&sm.tmem_base, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (tid < kTailMax) {
    int ps = -1;
    if (tid < n0) ps = __ldcg(p.pos + (static_cast<size_t>(l0) * B + b) * L + tid);
    sm.pos[0][tid] = ps;
    const uint32_t bits = __ballot_sync(0xffffffffu, tid < n0 && tail_is_global(sm, ps));
    if (lane == 0) sm.gbits[0][warp] = bits;
  }
  const uint32_t tm = sm.tmem_base;
  volatile int* abort_flag = &sm.abort;
  const uint32_t q_a = smem_u32(base), k_a = q_a + kTailOpBytes, v_a = k_a + kTailOpBytes;
  const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;

  uint32_t cnt0 = 0, cnt1 = 0;   // layers in which tile X (0, 1) was in use: barrier phases
  int cur = 0;
  for (int l = l0; l < n_layers; ++l) {
    const int it = l - l0;
    __syncthreads();   // sm.pos / sm.n / sm.gbits of this layer are complete
    const int n = sm.n[cur];
    const int nX = n > kTile ? 2 : 1;
    const int n16 = (n + 15) & ~15;
    const int nc2 = (n + 63) >> 6;     // 64-wide steps of a row (or column)
    const int par = it & 1;

    // ---- rows of the current tokens: 16-byte pieces, 128B-swizzled tiles
    {
      // thread tid copies 16-byte piece (tid & 7) of every 36th row, the
      // same piece of Q, K and V from one address computation
      const size_t tok0 = (static_cast<size_t>(l) * B + b) * L;
      const int piece = tid & 7;
      for (int r = tid >> 3; r < n; r += kTailThreads / 8) {
        const size_t off = ((tok0 + sm.pos[cur][r]) * H + h) * kHeadDim + 8 * piece;
        const uint32_t so = sw128_offset(r, piece);
        cp_async16(q_a + so, p.src[0] + off);
        cp_async16(k_a + so, p.src[1] + off);
        cp_async16(v_a + so, p.src[2] + off);
      }
      if (l + 1 < n_layers) {
        // the next layer's tokens are a subset of the current ones
        const size_t tok1 = (static_cast<size_t>(l + 1) * B + b) * L;
        for (int r = tid; r < n; r += kTailThreads) {
          const size_t off = ((tok1 + sm.pos[cur][r]) * H + h) * kHeadDim;
#pragma unroll
          for (int t = 0; t < 3; ++t) prefetch_l2_line(p.src[t] + off);
        }
      }
      cp_async_wait_all();
      fence_proxy_async_smem();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    if (warp == 8) {
      // ------------------------------------------------------- MMA issue
      if (lane == 0 && *abort_flag == 0) {
        const uint32_t id_s = idesc_bf16(128, n16, false, false);
        const uint32_t id_pv = idesc_bf16(128, 64, false, true);
        for (int X = 0; X < nX; ++X) {
#pragma unroll
          for (int k = 0; k < kHeadDim / 16; ++k)
            umma_bf16(tm + 256u * X, sdesc_sw128(q_a + X * kTileBytes + 32 * k),
                      sdesc_sw128(k_a + 32 * k), id_s, k > 0);
          umma_commit(&sm.bar_s[X]);
        }
        if (nX == 1) {
          // one query tile leaves the second half of tensor memory free: S^T
          // of the (single) key tile goes there at once
#pragma unroll
          for (int k = 0; k < kHeadDim / 16; ++k)
            umma_bf16(tm + 256u, sdesc_sw128(k_a + 32 * k), sdesc_sw128(q_a + 32 * k), id_s, k > 0);
          umma_commit(&sm.bar_st[0]);
        }
        bool ok = true;
        for (int X = 0; ok && X < nX; ++X) {
          if (!(ok = mbar_wait(&sm.bar_p[X], (X ? cnt1 : cnt0) & 1, abort_flag))) break;
          tc_fence_after();
          for (int k = 0; k < n16 / 16; ++k)
            umma_bf16_ts(tm + 256u * X + 128u, tm + 256u * X + 8u * k,
                         sdesc_sw128(v_a + 2048u * k), id_pv, k > 0);
          umma_commit(&sm.bar_o[X]);
        }
        // two query tiles: S^T of key tile X overwrites warpgroup X's columns
        // once that warpgroup has read its O
        for (int X = 0; ok && nX == 2 && X < 2; ++X) {
          if (!(ok = mbar_wait(&sm.bar_free[X], it & 1, abort_flag))) break;
          tc_fence_after();
#pragma unroll
          for (int k = 0; k < kHeadDim / 16; ++k)
            umma_bf16(tm + 256u * X, sdesc_sw128(k_a + X * kTileBytes + 32 * k),
                      sdesc_sw128(q_a + 32 * k), id_s, k > 0);
          umma_commit(&sm.bar_st[X]);
        }
      }
      __syncwarp();
    } else {
      // ------------------------------------------------------- softmax warps
      const int X = warp >> 2;
      const int i = kTile * X + (tid & 127);   // query row (rows step) / key column (cols step)
      const bool use = X < nX;
      const uint32_t ph = (X ? cnt1 : cnt0) & 1;
      const uint32_t tS = tm + 256u * X, tO = tS + 128u;
      Partners me;
      me.valid = i < n;
      me.lo = max(0, i - w);
      me.hi = min(n - 1, i + w);
      me.all = w >= n - 1 || ((sm.gbits[cur][i >> 5] >> (i & 31)) & 1u);
      float lse = INFINITY;
      if (use && tail_wait(&sm.bar_s[X], ph, abort_flag)) {
        tc_fence_after();
        // pass 1: row maximum over the allowed keys, 64 columns per step
        float pm[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
        for (int q2 = 0; q2 < nc2; ++q2) {
          float x[64];
          tmem_ld32(tS + lane_off + 64 * q2, x);
          tmem_ld32(tS + lane_off + 64 * q2 + 32, x + 32);
          tmem_ld_wait();
#pragma unroll
          for (int hq = 0; hq < 2; ++hq) {
            apply_mask(x + 32 * hq, partner_mask(me, sm, cur, 2 * q2 + hq, n));
#pragma unroll
            for (int k = 0; k < 32; ++k) pm[k & 3] = fmaxf(pm[k & 3], x[32 * hq + k]);
          }
        }
        const float mx = fmaxf(fmaxf(pm[0], pm[1]), fmaxf(pm[2], pm[3]));
        const float nmc = me.valid ? -mx * kLogitScale2 : 0.f;
        // pass 2: P = exp2(S - max) (masked keys: exp2(-inf) = 0), row sum, and
        // P as bf16 pairs over the first half of each step's columns (they
        // land in columns that this or earlier steps occupied, already read)
        const uint64_t c2 = f2_pack(kLogitScale2, kLogitScale2), n2 = f2_pack(nmc, nmc);
        uint64_t s2a = f2_pack(0.f, 0.f), s2b = s2a;
        for (int q2 = 0; q2 < nc2; ++q2) {
          float x[64];
          tmem_ld32(tS + lane_off + 64 * q2, x);
          tmem_ld32(tS + lane_off + 64 * q2 + 32, x + 32);
          tmem_ld_wait();
#pragma unroll
          for (int hq = 0; hq < 2; ++hq) {
            float* xh = x + 32 * hq;
            apply_mask(xh, partner_mask(me, sm, cur, 2 * q2 + hq, n));
            uint32_t pk[16];
#pragma unroll
            for (int k = 0; k < 32; k += 2) {
              float u, v;
              f2_unpack(f2_fma(f2_pack(xh[k], xh[k + 1]), c2, n2), u, v);
              u = ex2(u);
              v = ex2(v);
              if (k & 2) s2b = f2_add(s2b, f2_pack(u, v));
              else s2a = f2_add(s2a, f2_pack(u, v));
              pk[k >> 1] = pack_bf16x2(u, v);
            }
            tmem_st16(tS + lane_off + 32 * q2 + 16 * hq, pk);
          }
        }
        tmem_st_wait();
        float la, lb, lc, ld;
        f2_unpack(s2a, la, lb);
        f2_unpack(s2b, lc, ld);
        const float lsum = (la + lb) + (lc + ld);
        tc_fence_before();
        mbar_arrive(&sm.bar_p[X]);
        if (tail_wait(&sm.bar_o[X], ph, abort_flag)) {
          tc_fence_after();
          lse = me.valid ? lg2(lsum) - nmc : INFINITY;
          const float inv = me.valid ? 1.f / lsum : 0.f;
          uint16_t* orow =
              p.O + (((static_cast<size_t>(l) * B + b) * L + i) * H + h) * kHeadDim;
          float o[64];
          tmem_ld32(tO + lane_off, o);
          tmem_ld32(tO + lane_off + 32, o + 32);
          tmem_ld_wait();
          if (me.valid) {
#pragma unroll
            for (int k = 0; k < 64; k += 8) {
              const uint4 v = make_uint4(pack_bf16x2(o[k] * inv, o[k + 1] * inv),
                                         pack_bf16x2(o[k + 2] * inv, o[k + 3] * inv),
                                         pack_bf16x2(o[k + 4] * inv, o[k + 5] * inv),
                                         pack_bf16x2(o[k + 6] * inv, o[k + 7] * inv));
              *reinterpret_cast<uint4*>(orow + k) = v;
            }
          }
        }
      }
      // this warpgroup has read its S, P and O: with two query tiles its
      // columns take S^T of key tile X next
      tc_fence_before();
      mbar_arrive(&sm.bar_free[X]);
      sm.nlse[i] = -lse;
      tail_named_sync();   // every LSE is written

      // columns: key j = i of this thread, summed over the query rows
      float acc = 0.f;
      if (use && tail_wait(&sm.bar_st[X], ph, abort_flag)) {
        tc_fence_after();
        const uint32_t tST = nX == 1 ? tm + 256u : tS;
        const uint64_t c2 = f2_pack(kLogitScale2, kLogitScale2);
        uint64_t a2a = f2_pack(0.f, 0.f), a2b = a2a;
        for (int q2 = 0; q2 < nc2; ++q2) {
          float x[64];
          tmem_ld32(tST + lane_off + 64 * q2, x);
          tmem_ld32(tST + lane_off + 64 * q2 + 32, x + 32);
          tmem_ld_wait();
#pragma unroll
          for (int hq = 0; hq < 2; ++hq) {
            float* xh = x + 32 * hq;
            apply_mask(xh, partner_mask(me, sm, cur, 2 * q2 + hq, n));
            const float* lw = sm.nlse + 64 * q2 + 32 * hq;
#pragma unroll
            for (int k = 0; k < 32; k += 4) {
              const float4 l4 = *reinterpret_cast<const float4*>(lw + k);
              float e0, e1, e2, e3;
              f2_unpack(f2_fma(f2_pack(xh[k], xh[k + 1]), c2, f2_pack(l4.x, l4.y)), e0, e1);
              f2_unpack(f2_fma(f2_pack(xh[k + 2], xh[k + 3]), c2, f2_pack(l4.z, l4.w)), e2, e3);
              a2a = f2_add(a2a, f2_pack(ex2(e0), ex2(e1)));
              a2b = f2_add(a2b, f2_pack(ex2(e2), ex2(e3)));
            }
          }
        }
        float a0, a1, a2, a3;
        f2_unpack(a2a, a0, a1);
        f2_unpack(a2b, a2, a3);
        acc = (a0 + a2) + (a1 + a3);
      }
      if (use) sm.colsum[par][i] = acc;
    }

    // ------------------------------------------------- heads, threshold, compaction
    tc_fence_before();
    cluster_sync();
    tc_fence_after();
    const int nxt = cur ^ 1;
    if (tid < kTailMax) {
      const int j = tid;
      bool keep = false;
      if (j < n) {
        const uint32_t la = smem_u32(&sm.colsum[par][j]);
        float v[kTailMaxHeads];
#pragma unroll
        for (int hh = 0; hh < kTailMaxHeads; ++hh)
          v[hh] = hh < H ? ld_dsmem_f32(dsmem_addr(la, hh)) : 0.f;
        float a = 0.f;
#pragma unroll
        for (int hh = 0; hh < kTailMaxHeads; ++hh)
          if (hh < H) a += v[hh];
        const float s = a / static_cast<float>(H * n);
        keep = (j == 0) || (s >= p.alpha[l] / static_cast<float>(n));
        if (h == 0) p.scores[(static_cast<size_t>(l) * B + b) * L + j] = s;
      }
      const uint32_t kb = __ballot_sync(0xffffffffu, keep);
      if (lane == 0) sm.wcnt[warp] = __popc(kb);
      tail_named_sync();
      int off = 0, total = 0;
#pragma unroll
      for (int w8 = 0; w8 < 8; ++w8) {
        const int c = sm.wcnt[w8];
        off += (w8 < warp) ? c : 0;
        total += c;
      }
      if (keep) {
        const int k = off + __popc(kb & ((1u << lane) - 1u));
        const int ps = sm.pos[cur][j];
        sm.pos[nxt][k] = ps;
        if (h == 0) p.pos[(static_cast<size_t>(l + 1) * B + b) * L + k] = ps;
      }
      if (tid == 0) {
        sm.n[nxt] = total;
        if (h == 0) p.len[static_cast<size_t>(l + 1) * B + b] = total;
      }
      tail_named_sync();
      const bool gk = tid < total && tail_is_global(sm, sm.pos[nxt][tid]);
      const uint32_t gb = __ballot_sync(0xffffffffu, gk);
      if (lane == 0) sm.gbits[nxt][warp] = gb;
    }
    cnt0 += 1;
    cnt1 += (nX == 2) ? 1 : 0;
    cur = nxt;
  }

  // no CTA leaves while another may still read its column sums
  tc_fence_before();
  cluster_sync();
  if (warp == 8) {
    if (lane == 0) {
      // after an expired wait, MMAs may still be in flight
      umma_commit(&sm.bar_fin);
      int dummy = 0;
      mbar_wait(&sm.bar_fin, 0, &dummy, 1000000000ull);
    }
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tm, 512);
  }
  if (tid == 0 && sm.abort) atomicOr(p.status, kStatusTimeout);
}

// ---------------------------------------------------------------------------
// launch helpers used by the C ABI
// ---------------------------------------------------------------------------
cudaError_t configure_tail() {
  cudaError_t e = cudaFuncSetAttribute(sc_tail_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(kTailDyn));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(sc_tail_kernel, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
  return e;
}

static cudaLaunchConfig_t tail_config(int B, int H, cudaStream_t st, cudaLaunchAttribute* attr) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(B * H));
  cfg.blockDim = dim3(kTailThreads);
  cfg.dynamicSmemBytes = kTailDyn;
  cfg.stream = st;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(H);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cfg;
}

// Clusters of H CTAs of the tail kernel that the device can hold at once
// (0: this cluster shape cannot be scheduled).
cudaError_t tail_max_clusters(int H, int* out) {
  *out = 0;
  if (H < 1 || H > kTailMaxHeads) return cudaSuccess;
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = tail_config(1, H, nullptr, attr);
  return cudaOccupancyMaxActiveClusters(out, sc_tail_kernel, &cfg);
}

cudaError_t launch_tail(const TailParams& p, cudaStream_t st) {
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = tail_config(p.B, p.H, st, attr);
  return cudaLaunchKernelEx(&cfg, sc_tail_kernel, p);
}

}  // namespace sc
