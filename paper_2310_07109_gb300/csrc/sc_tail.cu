// sc_tail.cu -- the remaining layers of a sequence once at most 384 tokens
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
//   rows     per 128-row query tile: S = Q K^T over the keys in halves of at
//            most 256 (tensor memory), an exact two-pass softmax in fp32 (base
//            2), P (bf16) back to tensor memory, O = P V accumulated over the
//            halves, LSE_i
//   columns  per 128-key tile: S^T = K Q^T over the queries in halves, and per
//            key column j the sum over rows of exp2(S_ij - LSE_i): one thread
//            per column, no cross-thread sums
//   heads    each CTA writes its column sums into every CTA of the cluster
//            (distributed shared memory) before the cluster barrier; every CTA
//            then adds the heads in the same fixed order, so all
//            take the same keep decisions (s_j >= alpha_l / n, j == 0 kept) and
//            compact the token list the same way, without a second exchange
//
// Softmax warpgroup X takes query tiles X and X + 2 and key tiles X and X + 2;
// its own MMA-issuing thread serves it in a fixed order of events, so each
// tcgen05.commit covers that warpgroup's MMAs only.
//
// The allowed set (window, global tokens), the softmax, the vertical
// accumulation and the order-preserving removal are those of Sec. "Sparse
// Attention", Sec. "Extractor of Attention Scores in Sparse Attention Matrix"
// and Sec. "Token Pruning"; global rows are ordinary rows here (their whole row
// of at most 384 keys is evaluated).
#include <cuda_runtime.h>
#include <cstdint>

#include "sc_internal.cuh"
#include "sc_select.cuh"
#include "sm103_primitives.cuh"

namespace sc {

constexpr int kTailThreads = 320;   // 2 softmax warpgroups + 2 MMA-issuing warps
constexpr int kTailTiles = (kTailMax + kTile - 1) / kTile;   // 128-row tiles (3)
constexpr uint32_t kTailOpBytes = kTailTiles * kTileBytes;   // rows of one tensor (48 KB)
constexpr int kTailChunks = kTailMax / 32;                    // 32-token chunks (12)
static_assert(kTailMax <= 384, "a second key half must fit beside O in tensor memory");
constexpr uint32_t kTailStageBytes = 8 * 2048;                // O row staging, 2 KB per softmax warp
// column sums of every head, [layer parity][head][column], written by the
// CTA of that head into every CTA of the cluster
constexpr uint32_t kTailColBytes = 2 * kTailMaxHeads * kTailMax * 4;
// Q, K, V operands, the O staging and alignment; more than half of an SM's
// shared memory, so a second CTA never shares the SM (each holds all 512
// tensor-memory columns while it waits at cluster barriers: two CTAs of
// different clusters on one SM could otherwise wait on each other's allocation).
constexpr uint32_t kTailDyn = 3 * kTailOpBytes + kTailStageBytes + kTailColBytes + 1024;
static_assert(kTailDyn > 233472 / 2, "the tail kernel must occupy an SM alone");

struct TailSmem {
  uint64_t bar_sfull[2], bar_sfree[2], bar_pready[2], bar_odone[2], bar_stfull[2], bar_fin[2];
  uint32_t tmem_base;
  int abort;
  int n[2];
  alignas(16) uint32_t kbits[2][8];   // compaction: ballot of kept tokens per (round, warp)
  int gpos[kMaxGlobal];               // global positions (sorted), -1 past n_global
  uint32_t gbits[2][kTailChunks];     // global flags of the current / next token list
  int32_t pos[2][kTailMax];           // original positions of the current / next tokens
  alignas(16) float nlse[kTailMax];   // -LSE of each query row (-inf past n)
  SelectSmem sel;                     // top-ratio rule: the cut's histogram
  uint8_t tie[kTailMax];              // ... and the ranks of exact ties at the cut
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

struct TailSync {   // the 256 softmax threads
  __device__ __forceinline__ void operator()() const { tail_named_sync(); }
};

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

__device__ __forceinline__ int round16(int x) { return (x + 15) & ~15; }

__global__ void __launch_bounds__(kTailThreads, 1)
    sc_tail_kernel(const __grid_constant__ TailParams p) {
  // the successor may start once every CTA is past its own grid wait, so it
  // finds the kernels before this one complete (the export of the per-layer
  // results runs beside this kernel)
  pdl_wait();
  pdl_launch_dependents();
  const int H = p.H, w = p.w, L = p.L, B = p.B, n_layers = p.n_layers;
  const int h = static_cast<int>(blockIdx.x) % H, b = static_cast<int>(blockIdx.x) / H;
  // every CTA of the cluster reads the same values: the exits below are uniform
  const int l0 = __ldcg(p.tail_from + b);
  if (l0 >= n_layers) return;
  const int n0 = __ldcg(p.len + static_cast<size_t>(l0) * B + b);
  // where this kernel's results go: the device arrays, or the caller's host buffers
  const bool to_host = p.hlen != nullptr;
  int32_t* const out_len = to_host ? p.hlen : p.len;
  int32_t* const out_pos = to_host ? p.hpos : p.pos;
  float* const out_scores = to_host ? p.hscores : p.scores;
  uint16_t* const out_O = to_host ? p.hO : p.O;
  uint16_t* const out_O_last = to_host ? p.hO_last : p.O_last;
  if (n0 <= 0 || n0 > kTailMax) {
    if (h == 0 && threadIdx.x == 0) {
      if (n0 > kTailMax) atomicOr(p.status, kStatusInternal);
      else
        for (int l = l0; l < n_layers; ++l) out_len[static_cast<size_t>(l + 1) * B + b] = 0;
      if (to_host && n0 <= kTailMax) p.hlen[static_cast<size_t>(l0) * B + b] = max(n0, 0);
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
    for (int X = 0; X < 2; ++X) {
      mbar_init(&sm.bar_sfull[X], 1);
      mbar_init(&sm.bar_sfree[X], 4);   // one arrival per warp
      mbar_init(&sm.bar_pready[X], 4);
      mbar_init(&sm.bar_odone[X], 1);
      mbar_init(&sm.bar_stfull[X], 1);
      mbar_init(&sm.bar_fin[X], 1);
    }
    sm.abort = 0;
    sm.n[0] = n0;
    fence_mbar_init();
  }
  if (tid < kMaxGlobal) sm.gpos[tid] = tid < p.n_global ? p.global_pos[tid] : -1;
  if (to_host && h == 0 && tid == 0) p.hlen[static_cast<size_t>(l0) * B + b] = n0;
  if (warp == 8) tmem_alloc(&sm.tmem_base, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  for (int c = tid; c < kTailChunks * 32; c += kTailThreads) {
    int ps = -1;
    if (c < n0) ps = __ldcg(p.pos + (static_cast<size_t>(l0) * B + b) * L + c);
    // the entering layer's tokens go to the host buffers with the rest
    if (to_host && h == 0 && c < n0) p.hpos[(static_cast<size_t>(l0) * B + b) * L + c] = ps;
    if (c < kTailMax) sm.pos[0][c] = ps;
    const uint32_t bits = __ballot_sync(0xffffffffu, c < n0 && tail_is_global(sm, ps));
    if (lane == 0) sm.gbits[0][c >> 5] = bits;
  }
  // the CTAs write into each other's shared memory from the first layer on:
  // each announces that it runs here and waits for the others after its
  // first gather
  cluster_arrive_relaxed();
  const uint32_t tm = sm.tmem_base;
  volatile int* abort_flag = &sm.abort;
  const uint32_t q_a = smem_u32(base), k_a = q_a + kTailOpBytes, v_a = k_a + kTailOpBytes;
  float* const colall = reinterpret_cast<float*>(base + 3 * kTailOpBytes + kTailStageBytes);
  const uint32_t lane_off = static_cast<uint32_t>((warp & 3) * 32) << 16;
  const uint64_t c2 = f2_pack(kLogitScale2, kLogitScale2);

  // barrier phases consumed so far (kernel lifetime; both sides count alike)
  uint32_t n_sfull = 0, n_stfull = 0, n_odone = 0;   // softmax side
  uint32_t n_sfree = 0, n_ready = 0;                  // issuing side
  int cur = 0;
  for (int l = l0; l < n_layers; ++l) {
    const int it = l - l0;
    __syncthreads();   // sm.pos / sm.n / sm.gbits of this layer are complete
    const int n = sm.n[cur];
    const int nq = (n + kTile - 1) / kTile;   // 128-row tiles (1..3)
    const int nkh = n > 256 ? 2 : 1;          // key (query) halves of at most 256
    const int par = it & 1;

    // ---- rows of the current tokens: 16-byte pieces, 128B-swizzled tiles
    {
      // thread tid copies 16-byte piece (tid & 7) of every 40th row, the
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
      if (l + 1 < n_layers && !p.src_host) {
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
    if (it == 0) cluster_wait();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();

    if (warp >= 8) {
      // ------------------------------------------------------- MMA issue
      const int X = warp - 8;
      if (lane == 0 && X < nq && *abort_flag == 0) {
        const uint32_t tR = tm + 256u * X;              // this warpgroup's columns
        const uint32_t id_pv = idesc_bf16(128, 64, false, true);
        bool first = true, ok = true;
        // the warpgroup's columns may be overwritten: the previous contents are read
        auto region = [&]() -> bool {
          if (first) {
            first = false;
            return true;
          }
          return mbar_wait(&sm.bar_sfree[X], (n_sfree++) & 1, abort_flag);
        };
        auto ready = [&]() -> bool {
          return mbar_wait(&sm.bar_pready[X], (n_ready++) & 1, abort_flag);
        };
        auto issue_s = [&](int qt, int kh) {   // S of query tile qt against key half kh
          const int N = round16(min(256, n - 256 * kh));
          const uint32_t id = idesc_bf16(128, N, false, false);
          tc_fence_after();
#pragma unroll
          for (int k = 0; k < kHeadDim / 16; ++k)
            umma_bf16(tR, sdesc_sw128(q_a + qt * kTileBytes + 32 * k),
                      sdesc_sw128(k_a + kh * 2 * kTileBytes + 32 * k), id, k > 0);
          umma_commit(&sm.bar_sfull[X]);
        };
        auto issue_pv = [&](int kh, bool acc) {   // O (+)= P V over key half kh
          const int N = round16(min(256, n - 256 * kh));
          tc_fence_after();
          for (int k = 0; k < N / 16; ++k)
            umma_bf16_ts(tR + 128u, tR + 8u * k, sdesc_sw128(v_a + kh * 2 * kTileBytes + 2048u * k),
                         id_pv, (acc || k > 0) ? 1u : 0u);
          umma_commit(&sm.bar_odone[X]);
        };
        auto issue_st = [&](int kt, int qh, uint32_t dst) {   // S^T of key tile kt, query half qh
          const int N = round16(min(256, n - 256 * qh));
          const uint32_t id = idesc_bf16(128, N, false, false);
          tc_fence_after();
#pragma unroll
          for (int k = 0; k < kHeadDim / 16; ++k)
            umma_bf16(dst, sdesc_sw128(k_a + kt * kTileBytes + 32 * k),
                      sdesc_sw128(q_a + qh * 2 * kTileBytes + 32 * k), id, k > 0);
          umma_commit(&sm.bar_stfull[X]);
        };
        for (int r = 0; ok && r < 2; ++r) {
          const int qt = X + 2 * r;
          if (qt >= nq) break;
          if (nkh == 1) {
            if (!(ok = region())) break;
            issue_s(qt, 0);
            // one query tile: the other half of tensor memory takes S^T at once
            if (nq == 1) issue_st(0, 0, tm + 256u);
            if (!(ok = ready())) break;
            issue_pv(0, false);
          } else {
            if (!(ok = region())) break;
            issue_s(qt, 0);
            if (!(ok = ready())) break;
            issue_pv(0, false);
            // key half 1 has at most 128 columns: its S lands on P of half 0
            // (not on O) after that half's P V in issue order, so it may be
            // issued at once
            issue_s(qt, 1);
            if (!(ok = ready())) break;
            issue_pv(1, true);
          }
        }
        for (int r = 0; ok && nq > 1 && r < 2; ++r) {
          const int kt = X + 2 * r;
          if (kt >= nq) break;
          for (int qh = 0; ok && qh < nkh; ++qh) {
            if (!(ok = region())) break;
            issue_st(kt, qh, tR);
          }
        }
        if (ok) region();   // the last release of the layer
      }
      __syncwarp();
    } else {
      // ------------------------------------------------------- softmax warps
      const int X = warp >> 2;
      const int r = tid & 127;
      const uint32_t tR = tm + 256u * X + lane_off, tO = tR + 128u;
      bool ok = true;
      auto partners_of = [&](int i) {
        Partners me;
        me.valid = i < n;
        me.lo = max(0, i - w);
        me.hi = min(n - 1, i + w);
        me.all = w >= n - 1 || ((sm.gbits[cur][i >> 5] >> (i & 31)) & 1u);
        return me;
      };
      // row maximum over the keys of half kh (S in tensor memory)
      auto half_max = [&](const Partners& me, int kh, float mx) {
        const int nh = min(256, n - 256 * kh);
        for (int q2 = 0; q2 < (nh + 63) >> 6; ++q2) {
          float x[64];
          tmem_ld32(tR + 64 * q2, x);
          tmem_ld32(tR + 64 * q2 + 32, x + 32);
          tmem_ld_wait();
#pragma unroll
          for (int hq = 0; hq < 2; ++hq) {
            apply_mask(x + 32 * hq, partner_mask(me, sm, cur, 8 * kh + 2 * q2 + hq, n));
#pragma unroll
            for (int k = 0; k < 32; k += 2) mx = fmax3(mx, x[32 * hq + k], x[32 * hq + k + 1]);
          }
        }
        return mx;
      };
      // P = exp2(S - max) over half kh, written as bf16 pairs over the first
      // half of its columns (each step's pairs land on columns this or an
      // earlier step has read); returns the half's row sum
      // Returns the half's sum of the exponentials (fp32: the row's LSE, which
      // the column sums use) and adds to *osum the same values rounded to the
      // bf16 that P V multiplies (the normaliser of O, so that O is a weighted
      // mean of V rows whatever the rounding of P).
      auto half_exp = [&](const Partners& me, int kh, float nmc, float* osum) {
        const int nh = min(256, n - 256 * kh);
        const uint64_t n2 = f2_pack(nmc, nmc);
        uint64_t s2a = f2_pack(0.f, 0.f), s2b = s2a;
        float la = 0.f, lb = 0.f, lc = 0.f, ld = 0.f;
        for (int q2 = 0; q2 < (nh + 63) >> 6; ++q2) {
          float x[64];
          tmem_ld32(tR + 64 * q2, x);
          tmem_ld32(tR + 64 * q2 + 32, x + 32);
          tmem_ld_wait();
#pragma unroll
          for (int hq = 0; hq < 2; ++hq) {
            float* xh = x + 32 * hq;
            apply_mask(xh, partner_mask(me, sm, cur, 8 * kh + 2 * q2 + hq, n));
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
              if (k & 2) {
                lc = add_bf16_lo(lc, pk[k >> 1]);
                ld = add_bf16_hi(ld, pk[k >> 1]);
              } else {
                la = add_bf16_lo(la, pk[k >> 1]);
                lb = add_bf16_hi(lb, pk[k >> 1]);
              }
            }
            tmem_st16(tR + 32 * q2 + 16 * hq, pk);
          }
        }
        tmem_st_wait();
        *osum += (la + lb) + (lc + ld);
        float ea, eb, ec, ed;
        f2_unpack(s2a, ea, eb);
        f2_unpack(s2b, ec, ed);
        return (ea + eb) + (ec + ed);
      };
      auto release = [&]() {   // the warpgroup's columns are read
        tc_fence_before();
        warp_arrive(&sm.bar_sfree[X]);
      };

      // ---- rows: query tiles X and X + 2
      for (int rr = 0; ok && rr < 2; ++rr) {
        const int qt = X + 2 * rr;
        if (qt >= nq) break;
        const int i = kTile * qt + r;
        const Partners me = partners_of(i);
        if (!(ok = tail_wait(&sm.bar_sfull[X], (n_sfull++) & 1, abort_flag))) break;
        tc_fence_after();
        // half 0: P = exp2(S - max of half 0), exact when there is one half
        const float m0 = half_max(me, 0, -INFINITY);
        const float nmc0 = (me.valid && m0 != -INFINITY) ? -m0 * kLogitScale2 : 0.f;
        float nmc = nmc0;
        float osum = 0.f;
        float lsum = half_exp(me, 0, nmc0, &osum);
        tc_fence_before();
        warp_arrive(&sm.bar_pready[X]);
        if (nkh == 2) {
          // half 1 (at most 128 keys; its S lands on P of half 0 after that
          // half's P V, so O of half 0 is complete once S is): the reference
          // rises to its maximum when that exceeds the reference by more than
          // 8 (base 2, P below 2^8 otherwise), and O and the row sum are
          // rescaled exactly
          if (!(ok = tail_wait(&sm.bar_sfull[X], (n_sfull++) & 1, abort_flag))) break;
          if (!(ok = tail_wait(&sm.bar_odone[X], (n_odone++) & 1, abort_flag))) break;
          tc_fence_after();
          const float m1 = half_max(me, 1, -INFINITY);
          const bool raise = me.valid && m1 != -INFINITY &&
                             (m0 == -INFINITY || (m1 - m0) * kLogitScale2 > 8.f);
          float f = 1.f;
          if (raise) {
            f = m0 == -INFINITY ? 0.f : ex2((m0 - m1) * kLogitScale2);
            nmc = -m1 * kLogitScale2;
            lsum *= f;
            osum *= f;
          }
          if (__any_sync(0xffffffffu, raise)) {
#pragma unroll 1
            for (int c = 0; c < 64; c += 16) {
              float o[16];
              tmem_ld16(tO + c, o);
              tmem_ld_wait();
#pragma unroll
              for (int k = 0; k < 16; ++k) o[k] *= f;
              tmem_st16(tO + c, reinterpret_cast<const uint32_t*>(o));
              tmem_st_wait();   // o is reused
            }
          }
          lsum += half_exp(me, 1, nmc, &osum);
          tc_fence_before();
          warp_arrive(&sm.bar_pready[X]);
        }
        if (!(ok = tail_wait(&sm.bar_odone[X], (n_odone++) & 1, abort_flag))) break;
        tc_fence_after();
        const float inv = me.valid ? 1.f / osum : 0.f;
        float o[64];
        tmem_ld32(tO, o);
        tmem_ld32(tO + 32, o + 32);
        tmem_ld_wait();
        sm.nlse[i] = me.valid ? -(lg2(lsum) - nmc) : -INFINITY;
        // O is in registers: the columns may take S^T while O is stored
        release();
        // the warp's 32 rows leave in two column halves of 64 bytes (no O
        // but the last layer's when O is not kept)
        uint8_t* stage = base + 3 * kTailOpBytes + warp * 2048;
        uint16_t* const Ol = out_O != nullptr ? out_O + static_cast<size_t>(l) * B * L * H * kHeadDim
                             : l == n_layers - 1 ? out_O_last : nullptr;
        uint16_t* row0 =
            Ol ? Ol + ((static_cast<size_t>(b) * L + i - (r & 31)) * H + h) * kHeadDim : nullptr;
        const uint32_t rows = __ballot_sync(0xffffffffu, me.valid);
#pragma unroll
        for (int c = 0; c < 64 && Ol != nullptr; c += 32) {
#pragma unroll
          for (int k = 0; k < 32; k += 8)
            stage_row_piece<4>(stage, k >> 3,
                               make_uint4(pack_bf16x2(o[c + k] * inv, o[c + k + 1] * inv),
                                          pack_bf16x2(o[c + k + 2] * inv, o[c + k + 3] * inv),
                                          pack_bf16x2(o[c + k + 4] * inv, o[c + k + 5] * inv),
                                          pack_bf16x2(o[c + k + 6] * inv, o[c + k + 7] * inv)));
          flush_staged_rows<4>(stage, row0 + c, static_cast<size_t>(H) * kHeadDim, rows);
        }
      }
      // rows past the last query tile take no part in the column sums
      for (int i = kTile * nq + (tid & 255); i < kTailMax; i += 256) sm.nlse[i] = -INFINITY;
      tail_named_sync();   // every LSE is written

      // ---- columns: key tiles X and X + 2, summed over the query rows
      for (int rr = 0; ok && rr < 2; ++rr) {
        const int kt = X + 2 * rr;
        if (kt >= nq) break;
        const int j = kTile * kt + r;
        const Partners me = partners_of(j);
        const uint32_t tST = nq == 1 ? tm + 256u + lane_off : tR;
        uint64_t a2a = f2_pack(0.f, 0.f), a2b = a2a;
        for (int qh = 0; ok && qh < nkh; ++qh) {
          if (!(ok = tail_wait(&sm.bar_stfull[X], (n_stfull++) & 1, abort_flag))) break;
          tc_fence_after();
          const int nh = min(256, n - 256 * qh);
          for (int q2 = 0; q2 < (nh + 63) >> 6; ++q2) {
            float x[64];
            tmem_ld32(tST + 64 * q2, x);
            tmem_ld32(tST + 64 * q2 + 32, x + 32);
            tmem_ld_wait();
#pragma unroll
            for (int hq = 0; hq < 2; ++hq) {
              const int qa = 8 * qh + 2 * q2 + hq;   // chunk of query rows
              float* xh = x + 32 * hq;
              apply_mask(xh, partner_mask(me, sm, cur, qa, n));
              const float* lw = sm.nlse + 32 * qa;
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
          if (nq > 1) release();
        }
        float a0, a1, a2, a3;
        f2_unpack(a2a, a0, a1);
        f2_unpack(a2b, a2, a3);
        // this head's sum of column j goes to every CTA of the cluster; the
        // cluster barrier below (release / acquire) makes it visible there
        const float cs = me.valid ? (a0 + a2) + (a1 + a3) : 0.f;
        const uint32_t la = smem_u32(colall + (par * kTailMaxHeads + h) * kTailMax + j);
        for (int hh = 0; hh < H; ++hh) st_dsmem_f32(dsmem_addr(la, hh), cs);
      }
    }

    // ------------------------------------------------- heads, threshold, compaction
    tc_fence_before();
    cluster_sync();
    tc_fence_after();
    const int nxt = cur ^ 1;
    if (tid < 256) {
      float sj[2] = {0.f, 0.f};
#pragma unroll
      for (int rd = 0; rd < 2; ++rd) {
        const int j = tid + 256 * rd;
        if (j < n) {
          const float* cj = colall + par * kTailMaxHeads * kTailMax + j;
          float v[kTailMaxHeads];
#pragma unroll
          for (int hh = 0; hh < kTailMaxHeads; ++hh) v[hh] = hh < H ? cj[hh * kTailMax] : 0.f;
          float a = 0.f;
#pragma unroll
          for (int hh = 0; hh < kTailMaxHeads; ++hh)
            if (hh < H) a += v[hh];
          sj[rd] = a / static_cast<float>(H * n);
          if (h == 0) out_scores[(static_cast<size_t>(l) * B + b) * L + j] = sj[rd];
        }
      }
      // keep flags: the threshold (relative or absolute), or the top-ratio cut
      // over the n scores (every CTA of the cluster finds the same cut)
      bool keep[2];
      if (p.keep_rule == kKeepTopRatio) {
        uint32_t key[2];
#pragma unroll
        for (int rd = 0; rd < 2; ++rd) {
          const int j = tid + 256 * rd;
          key[rd] = (j >= 1 && j < n) ? select_key(sj[rd]) : 0u;
        }
        uint32_t cut;
        int ties, eq;
        radix_cut<256, 2>(key, top_count(p.alpha[l], n) - 1, n - 1, sm.sel, tid, TailSync(), cut,
                          ties, eq);
        const bool split = eq > ties;
        if (split) rank_ties<256, 2>(key, cut, ties, n, sm.tie, tid, TailSync());
#pragma unroll
        for (int rd = 0; rd < 2; ++rd) {
          const int j = tid + 256 * rd;
          keep[rd] = j < n && (j == 0 || key[rd] > cut ||
                               (key[rd] == cut && (!split || sm.tie[j] == 2)));
        }
      } else {
        const float thr = p.keep_rule == kKeepAbsolute ? p.alpha[l]
                                                       : p.alpha[l] / static_cast<float>(n);
#pragma unroll
        for (int rd = 0; rd < 2; ++rd) {
          const int j = tid + 256 * rd;
          keep[rd] = j < n && (j == 0 || sj[rd] >= thr);
        }
      }
#pragma unroll
      for (int rd = 0; rd < 2; ++rd) {
        const uint32_t kb = __ballot_sync(0xffffffffu, keep[rd]);
        if (lane == 0) sm.kbits[rd][warp] = kb;
      }
      tail_named_sync();
      // every thread reads the 16 ballot words (round-major, then warp) and
      // forms its own exclusive prefix and the total
      int kpre[2] = {0, 0}, total = 0;
      {
        const uint4* kw = reinterpret_cast<const uint4*>(&sm.kbits[0][0]);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const uint4 u = kw[q];
          const uint32_t wv[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const int idx = 4 * q + e;   // = 8 * round + warp
            if (idx == warp) kpre[0] = total;
            if (idx == 8 + warp) kpre[1] = total;
            total += __popc(wv[e]);
          }
        }
      }
#pragma unroll
      for (int rd = 0; rd < 2; ++rd) {
        if (!keep[rd]) continue;
        const int j = tid + 256 * rd;
        const int k = kpre[rd] + __popc(sm.kbits[rd][warp] & ((1u << lane) - 1u));
        const int ps = sm.pos[cur][j];
        sm.pos[nxt][k] = ps;
        if (h == 0) out_pos[(static_cast<size_t>(l + 1) * B + b) * L + k] = ps;
      }
      if (tid == 0) {
        sm.n[nxt] = total;
        if (h == 0) out_len[static_cast<size_t>(l + 1) * B + b] = total;
      }
      tail_named_sync();
#pragma unroll
      for (int rd = 0; rd < 2; ++rd) {
        const int k = tid + 256 * rd;
        const bool gk = k < total && tail_is_global(sm, sm.pos[nxt][k]);
        const uint32_t gb = __ballot_sync(0xffffffffu, gk);
        if (lane == 0 && (k >> 5) < kTailChunks) sm.gbits[nxt][k >> 5] = gb;
      }
    }
    cur = nxt;
  }

  // no CTA leaves while another may still read its column sums
  tc_fence_before();
  cluster_sync();
  if (warp >= 8 && warp - 8 < 2) {
    if (lane == 0) {
      // after an expired wait, MMAs may still be in flight
      umma_commit(&sm.bar_fin[warp - 8]);
      int dummy = 0;
      mbar_wait(&sm.bar_fin[warp - 8], 0, &dummy, 1000000000ull);
    }
    __syncwarp();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 8) {
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
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = tail_config(p.B, p.H, st, attr);
  // chained like the per-layer kernels: scheduled while its predecessor
  // finishes, waiting for it on the device
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, sc_tail_kernel, p);
}

}  // namespace sc
