// sc_band.cu -- the single-pass rows kernel of one sparse-attention layer
// (windows up to 256 tokens on each side): every band tile's S = Q K^T is
// computed and exponentiated once.
//
// The column sums of Sec. "Pruning" (probabilities "accumulated vertically",
// Fig. 1) need each row's final normaliser, which is known only after the
// row's whole band.  Instead of a second pass that recomputes S^T and its
// exponentials, the kernel keeps every band tile's bf16 probabilities
// P~_t = 2^(x - m_t) (m_t the row's running reference when tile t was taken)
// in its own tensor-memory slot.  Once the row is complete, each row's weight
// c_{i,t} = 2^(m_t - LSE_i) turns P~_t into the normalised P_t, and the sums
// down the key columns are one tensor-core product per tile:
//     colsum_t[j] = sum_i P~_t[i, j] c_{i,t}    (M = 128 keys, N = 16, K = 128 rows)
// with P~_t^T read from shared memory in MN-major form and c as two bf16 terms
// (c_hi + c_lo) in the N columns 2t, 2t + 1 of a small weight matrix.  O is
// normalised by the sum of the same rounded probabilities (so O is a weighted
// mean of V rows whatever the rounding of P).
//
// Persistent: one CTA per SM walks query tiles (sequence, head)-major.  One
// 128-row query tile fills the SM's 512 tensor-memory columns
// (O 64 | S 128 | five 64-column slots of P~), so consecutive tiles overlap
// instead: the epilogue of tile k (O out, P~ staged for the column-sum
// products, sums out) runs on the helper warps while the softmax warps
// already work through tile k + 1, each slot handed back as soon as its
// column sums have been read.  The global keys of a row (Sec. "Extractor of
// Attention Scores": global tokens attend and are attended everywhere) join
// the row's softmax after its band, as one more 16-key block.
//
// Warps: 0-7 softmax (warp w: rows 32 (w & 3) .. + 31 = its tensor-memory
// lanes, keys 64 (w >> 2) .. + 63 of each band tile; the two warps of a row
// block share the row's running reference through shared memory), 8-11
// helpers (the previous tile's epilogue), 12 loads Q, the global rows and the
// K ring, 13 issues the S and P V products, 14 loads the V ring, 15 holds the
// tensor memory and issues the column-sum products.  Its outputs are those of
// the paired rows kernel (O, the band rows' column sums per query tile, the
// global keys' far-row sums, the global queries' (max, sum) pieces), so the
// cols kernel is the same for both.
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cstdint>

#include "sc_internal.cuh"
#include "sc_layer_common.cuh"
#include "sm103_primitives.cuh"

namespace sc {

constexpr int kBandThreads = 512;
constexpr int kBandSoftmaxRegs = 168;
constexpr int kBandHelperRegs = 120;
constexpr int kBandCtlRegs = 56;
// warpgroups: two softmax, helpers, control (launched with 128 a thread)
static_assert(256 * kBandSoftmaxRegs + 128 * kBandHelperRegs + 128 * kBandCtlRegs <= 65536,
              "register split exceeds the launch allocation");
constexpr int kBandKStages = 3;
constexpr int kBandVStages = 3;
constexpr uint32_t kStageBytes = 2 * kTileBytes;   // one 128 x 128 bf16 tile
constexpr int kNoSlot = kMaxBandTiles;             // index of the global block's P V

// tensor memory columns
constexpr uint32_t kColO = 0;
constexpr uint32_t kColS = 64;          // S_t; also S_Gt, S_G (16) and P_G (8, at +16)
constexpr uint32_t kColPG = kColS + 16;
__host__ __device__ constexpr uint32_t col_slot(int t) { return 192u + 64u * t; }
static_assert(col_slot(kMaxBandTiles) == 512, "the slots end at the last column");

// dynamic shared memory (1024-byte aligned base)
constexpr uint32_t kOffQ = 0;                                      // two Q tiles
constexpr uint32_t kOffK = kOffQ + 2 * kTileBytes;
constexpr uint32_t kOffV = kOffK + kBandKStages * kTileBytes;
constexpr uint32_t kOffStage = kOffV + kBandVStages * kTileBytes;  // two staging tiles
constexpr uint32_t kOffG = kOffStage + 2 * kStageBytes;            // two sets: K_G, Q_G, V_G
constexpr uint32_t kGSetBytes = 3 * kGTileBytes;
constexpr uint32_t kOffW = kOffG + 2 * kGSetBytes;                 // two weight matrices
constexpr uint32_t kWBytes = 16 * kTile * 2;                       // [16][128] bf16
constexpr uint32_t kBandDyn = kOffW + 2 * kWBytes + 1024;
static_assert(kOffStage % 1024 == 0 && kOffW % 1024 == 0 && kOffG % 1024 == 0 &&
              kGSetBytes % 1024 == 0, "swizzled operands start on 1024-byte boundaries");
static_assert(kBandDyn <= 227 * 1024 - 8 * 1024, "shared memory");

struct BandSmem {
  uint64_t bar_q[2], bar_qfree[2];
  uint64_t bar_kfull[kBandKStages], bar_kempty[kBandKStages];
  uint64_t bar_vfull[kBandVStages], bar_vempty[kBandVStages];
  uint64_t bar_sfull, bar_sfree;   // one product at a time in the S columns
  uint64_t bar_pready[2];          // P~ stored, alternating by P index
  uint64_t bar_pgready;            // P_G stored (half-0 softmax warps)
  uint64_t bar_pvdone[kMaxBandTiles + 1];   // P V of each slot, then of the global block
  uint64_t bar_pair[4];            // the two softmax warps of a row block
  uint64_t bar_epi;                // a tile's weights, 1/osum, O complete
  uint64_t bar_ofree;              // the helpers have read O
  uint64_t bar_stfull[2], bar_stfree[2];
  uint64_t bar_dfull[kMaxBandTiles];
  uint64_t bar_slotfree[kMaxBandTiles];
  uint64_t bar_fin, bar_fin2, bar_stall;
  uint32_t tmem_base;
  int abort;
  float xmax[2][2][kTile];         // [tile parity][half][row] partial maxima
  float xsum[2][2][2][kTile];      // [item parity][half][lsum, osum][row]
  float inv_osum[2][kTile];        // [item parity][row], 0 for rows without results
};

// One work item: query tile q of (sequence b, head h).
struct BandItem {
  int b, h, q, n, ng, klo, nk, diag;
  bool run;
};

__device__ __forceinline__ BandItem band_item(const LayerParams& p, const LayerView& v, int it) {
  BandItem x;
  const int bh = it / p.T;
  x.q = it - bh * p.T;
  x.h = bh % p.H;
  x.b = bh / p.H;
  x.run = false;
  x.n = x.ng = x.klo = x.nk = x.diag = 0;
  if (owned_by_tail(p, v, x.b)) return x;
  x.n = __ldcg(v.len + x.b);
  if (x.q * kTile >= x.n) return x;
  x.ng = min(__ldcg(v.ng + x.b), kMaxGlobal);
  const int q0 = x.q * kTile, q1 = min(q0 + kTile - 1, x.n - 1);
  x.klo = max(0, q0 - p.w) / kTile;
  x.nk = min(x.n - 1, q1 + p.w) / kTile - x.klo + 1;
  x.diag = x.q - x.klo;
  x.run = true;
  return x;
}

// 32 lanes x 2 consecutive 32-bit columns.
__device__ __forceinline__ void tmem_ld2(uint32_t taddr, float& a, float& b) {
  uint32_t r0, r1;
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x2.b32 {%0, %1}, [%2];"
               : "=r"(r0), "=r"(r1)
               : "r"(taddr));
  a = __uint_as_float(r0);
  b = __uint_as_float(r1);
}

// D[128 keys x 16] = A[128 keys x 128 rows] * W[128 rows x 16]: A is P~ of one
// key tile read transposed (MN-major: the 128-byte lines are rows of P~,
// 64-key atoms 1024 bytes apart, groups of 8 rows 2048 bytes apart), W the
// per-row weights (K-major [16][128], 64-row chunks 2048 bytes apart).
__device__ __forceinline__ void mma_colsum(uint32_t d_tmem, uint32_t a_smem, uint32_t w_smem) {
  const uint32_t idesc = idesc_bf16(128, 16, true, false);
#pragma unroll
  for (int k = 0; k < kTile / 16; ++k)
    umma_bf16(d_tmem, sdesc_sw128(a_smem + k * 4096, 2048, 1024),
              sdesc_sw128(w_smem + (k >> 2) * 2048 + (k & 3) * 32, 1024), idesc, k > 0 ? 1u : 0u);
}

// Byte offset of element (n, k) of the weight matrix [16][128] (K-major, 128B swizzle).
__device__ __forceinline__ uint32_t w_offset(int n, int k) {
  return (k >> 6) * 2048 + (n >> 3) * 1024 + sw128_offset(n & 7, (k & 63) >> 3) + (k & 7) * 2;
}

// Byte offset of the 16-byte chunk c (keys 8c .. 8c+7 of atom a) of row r in a
// staging tile of P~ (MN-major for the column-sum product, see mma_colsum).
__device__ __forceinline__ uint32_t stage_offset_mn(int r, int a, int c) {
  return (r >> 3) * 2048 + a * 1024 + sw128_offset(r & 7, c);
}

// Barrier over the four helper warps (id 3) whose outcome is the OR of every
// thread's `pred`: all of them take the same branch afterwards.
__device__ __forceinline__ bool helpers_sync_or(bool pred) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, 3, 128, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(pred ? 1u : 0u)
      : "memory");
  return r != 0;
}

// The (max, sum) of each global query over this warp's 32 keys of a key tile
// (lane = key; xt the 16 raw logits), for the cols kernel to merge into the
// global rows' normalisers.
__device__ __forceinline__ void global_query_stats(const LayerParams& p, const BandItem& x,
                                                   int wq, int r, const float (&xt)[kMaxGlobal]) {
  const int lane = threadIdx.x & 31;
  const bool key_ok = x.q * kTile + r < x.n;
  float y[kMaxGlobal], e16[kMaxGlobal];
#pragma unroll
  for (int g = 0; g < kMaxGlobal; ++g) {
    y[g] = (key_ok && g < x.ng) ? xt[g] * kLogitScale2 : -INFINITY;
    e16[g] = y[g];
  }
  const float mme = warp_reduce16(e16, OpMax());
#pragma unroll
  for (int g = 0; g < kMaxGlobal; ++g) {
    const float mg = __shfl_sync(0xffffffffu, mme, 2 * g);
    e16[g] = mg == -INFINITY ? 0.f : ex2(y[g] - mg);
  }
  const float sme = warp_reduce16(e16, OpAdd());
  const int gme = lane >> 1;
  const size_t slot0 = (((static_cast<size_t>(x.b) * p.H + x.h) * p.T + x.q) * 4 + wq) * kMaxGlobal;
  if ((lane & 1) == 0 && gme < x.ng) {
    p.gstat[2 * (slot0 + gme)] = mme;
    p.gstat[2 * (slot0 + gme) + 1] = sme;
  }
}

// Exponentials of one half tile (64 keys): P~ = 2^(x * scale - m) packed to
// bf16 pairs and stored to the tensor-memory columns at `taddr` (32 columns),
// one 32-key chunk at a time; the sums of the values (lsum, fp32) and of their
// bf16 roundings (osum).  Chunks of 32 keys that no row of the warp attends
// to take no exponentials.
__device__ __forceinline__ void exp_half_tile(const float (&xs)[64], float nref, bool alive0,
                                              bool alive1, uint32_t taddr, float& lsum,
                                              float& osum) {
  const uint64_t c2 = f2_pack(kLogitScale2, kLogitScale2);
  const uint64_t n2 = f2_pack(nref, nref);
  uint64_t s2a = f2_pack(0.f, 0.f), s2b = s2a;
  float sq[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
  for (int ch = 0; ch < 2; ++ch) {
    uint32_t pk[16];
    if (ch == 0 ? alive0 : alive1) {
#pragma unroll
      for (int k = 0; k < 32; k += 2) {
        float u, w;
        f2_unpack(f2_fma(f2_pack(xs[32 * ch + k], xs[32 * ch + k + 1]), c2, n2), u, w);
        u = ex2(u);
        w = ex2(w);
        if (k & 2) s2b = f2_add(s2b, f2_pack(u, w));
        else s2a = f2_add(s2a, f2_pack(u, w));
        pk[k >> 1] = pack_bf16x2(u, w);
        const int c = (k >> 1) & 1;
        sq[2 * c] = add_bf16_lo(sq[2 * c], pk[k >> 1]);
        sq[2 * c + 1] = add_bf16_hi(sq[2 * c + 1], pk[k >> 1]);
      }
    } else {
#pragma unroll
      for (int k = 0; k < 16; ++k) pk[k] = 0u;
    }
    tmem_st16(taddr + 16 * ch, pk);
  }
  float sa, sb, sc, sd;
  f2_unpack(s2a, sa, sb);
  f2_unpack(s2b, sc, sd);
  lsum += (sa + sb) + (sc + sd);
  osum += (sq[0] + sq[1]) + (sq[2] + sq[3]);
}

// Scale this warp's 32 O columns (the half `hf` of the row's 64) by f.
__device__ __forceinline__ void rescale_o(uint32_t taddr, float f) {
#pragma unroll 1
  for (int c = 0; c < 32; c += 16) {
    float o[16];
    tmem_ld16(taddr + c, o);
    tmem_ld_wait();
#pragma unroll
    for (int k = 0; k < 16; ++k) o[k] *= f;
    tmem_st16(taddr + c, reinterpret_cast<const uint32_t*>(o));
    tmem_st_wait();   // o is reused
  }
}

__global__ void __launch_bounds__(kBandThreads, 1)
    sc_band_kernel(const __grid_constant__ TensorMaps maps, const __grid_constant__ LayerParams p) {
  // the cols kernel is scheduled once every CTA here has passed this wait
  pdl_wait();
  pdl_launch_dependents();
  const LayerView v = layer_view(p);
  const int n_items = p.B * p.H * p.T;

  extern __shared__ uint8_t dyn_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dyn_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  __shared__ BandSmem sm;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  if (tid == 0) {
    for (int u = 0; u < 2; ++u) {
      mbar_init(&sm.bar_q[u], 1);
      mbar_init(&sm.bar_qfree[u], 1);
      mbar_init(&sm.bar_pready[u], 8);   // softmax warps
      mbar_init(&sm.bar_stfull[u], 4);   // helper warps
      mbar_init(&sm.bar_stfree[u], 1);
    }
    for (int s = 0; s < kBandKStages; ++s) {
      mbar_init(&sm.bar_kfull[s], 1);
      mbar_init(&sm.bar_kempty[s], 1);
    }
    for (int s = 0; s < kBandVStages; ++s) {
      mbar_init(&sm.bar_vfull[s], 1);
      mbar_init(&sm.bar_vempty[s], 1);
    }
    mbar_init(&sm.bar_sfull, 1);
    mbar_init(&sm.bar_sfree, 8);
    mbar_init(&sm.bar_pgready, 4);   // softmax warps of half 0
    for (int u = 0; u <= kMaxBandTiles; ++u) mbar_init(&sm.bar_pvdone[u], 1);
    for (int u = 0; u < 4; ++u) mbar_init(&sm.bar_pair[u], 2);
    mbar_init(&sm.bar_epi, 8);
    mbar_init(&sm.bar_ofree, 4);
    for (int t = 0; t < kMaxBandTiles; ++t) {
      mbar_init(&sm.bar_dfull[t], 1);
      mbar_init(&sm.bar_slotfree[t], 4);
    }
    mbar_init(&sm.bar_fin, 1);
    mbar_init(&sm.bar_fin2, 1);
    mbar_init(&sm.bar_stall, 1);
    sm.abort = 0;
    fence_mbar_init();
  }
  if (warp == 15) tmem_alloc(&sm.tmem_base, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = sm.tmem_base;
  volatile int* abort_flag = &sm.abort;

  if (warp >= 12) {
    regs_dealloc<kBandCtlRegs>();
    if (warp == 12) {
      // ------------------------------------------- Q and the global rows (two buffers), K ring
      uint32_t kc = 0, qn = 0;
      bool ok = true;
      for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x) {
        const BandItem x = band_item(p, v, it);
        if (!x.run) continue;
        const RowSource rs = row_source(p, v, x.b);
        const int qb = qn & 1;
        const int ngp = x.ng > 0 ? kMaxGlobal : 0;
        // this buffer is free once the products of the item two back are
        if (lane == 0 && qn >= 2) ok = mbar_wait(&sm.bar_qfree[qb], ((qn >> 1) - 1) & 1, abort_flag);
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        if (!ok) break;
        uint8_t* gset = base + kOffG + qb * kGSetBytes;
        if (lane == 0) {
          mbar_arrive_expect_tx(&sm.bar_q[qb], kTileBytes + 3 * ngp * 128);
          load_tile(maps, 0, rs, x.h, x.q * kTile, base + kOffQ + qb * kTileBytes, &sm.bar_q[qb]);
        }
        __syncwarp();
        if (ngp && lane < 4) {
          // lanes 0..3 gather four of the 16 global rows each (the last repeated)
          const int32_t* gcur = v.gcur + x.b * kMaxGlobal;
          int rr[4];
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int g = min(4 * lane + k, x.ng - 1);
            rr[k] = static_cast<int>((rs.tok_b + __ldcg(gcur + g)) * p.H + x.h);
          }
          // K_G, Q_G, V_G
          tma_gather4(gset + 512 * lane, &maps.row[rs.s][1], 0, rr[0], rr[1], rr[2], rr[3],
                      &sm.bar_q[qb]);
          tma_gather4(gset + kGTileBytes + 512 * lane, &maps.row[rs.s][0], 0, rr[0], rr[1], rr[2],
                      rr[3], &sm.bar_q[qb]);
          tma_gather4(gset + 2 * kGTileBytes + 512 * lane, &maps.row[rs.s][2], 0, rr[0], rr[1],
                      rr[2], rr[3], &sm.bar_q[qb]);
        }
        ++qn;
        if (lane == 0) {
          for (int t = 0; t < x.nk; ++t) {
            const int s = kc % kBandKStages;
            if (kc >= kBandKStages &&
                !(ok = mbar_wait(&sm.bar_kempty[s], (kc / kBandKStages - 1) & 1, abort_flag)))
              break;
            mbar_arrive_expect_tx(&sm.bar_kfull[s], kTileBytes);
            load_tile(maps, 1, rs, x.h, (x.klo + t) * kTile, base + kOffK + s * kTileBytes,
                      &sm.bar_kfull[s]);
            ++kc;
          }
        }
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
      }
      // nothing may still be landing in shared memory when the CTA exits
      if (lane == 0) {
        for (uint32_t s = 0; s < kBandKStages && s < kc; ++s) {
          const uint32_t last = s + kBandKStages * ((kc - 1 - s) / kBandKStages);
          drain_wait(&sm.bar_kfull[s], (last / kBandKStages) & 1);
        }
        for (uint32_t qb = 0; qb < 2 && qb < qn; ++qb) {
          const uint32_t uses = (qn - qb + 1) / 2;
          drain_wait(&sm.bar_q[qb], (uses - 1) & 1);
        }
      }
      __syncwarp();
    } else if (warp == 14) {
      // ------------------------------------------- V ring
      if (lane == 0) {
        uint32_t vc = 0;
        bool ok = true;
        for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x) {
          const BandItem x = band_item(p, v, it);
          if (!x.run) continue;
          const RowSource rs = row_source(p, v, x.b);
          for (int t = 0; t < x.nk; ++t) {
            const int s = vc % kBandVStages;
            if (vc >= kBandVStages &&
                !(ok = mbar_wait(&sm.bar_vempty[s], (vc / kBandVStages - 1) & 1, abort_flag)))
              break;
            mbar_arrive_expect_tx(&sm.bar_vfull[s], kTileBytes);
            load_tile(maps, 2, rs, x.h, (x.klo + t) * kTile, base + kOffV + s * kTileBytes,
                      &sm.bar_vfull[s]);
            ++vc;
          }
        }
        for (uint32_t s = 0; s < kBandVStages && s < vc; ++s) {
          const uint32_t last = s + kBandVStages * ((vc - 1 - s) / kBandVStages);
          drain_wait(&sm.bar_vfull[s], (last / kBandVStages) & 1);
        }
      }
      __syncwarp();
    } else if (warp == 13) {
      // ------------------------------------------- S and P V products
      if (lane == 0) {
        const uint32_t k_a = smem_u32(base + kOffK), v_a = smem_u32(base + kOffV);
        bool ok = true;
        if (p.stall_ns != 0)   // test hook: this bounded wait expires
          ok = mbar_wait(&sm.bar_stall, 0, abort_flag, p.stall_ns);
        uint32_t kc = 0, vc = 0, s_uses = 0, n_p = 0, item_no = 0, n_glob = 0;
        bool pg_pending = false;   // the previous item's P_G V_G reads the S columns
        for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x) {
          const BandItem x = band_item(p, v, it);
          if (!x.run) continue;
          const bool glob = x.ng > 0;
          const int qb = item_no & 1;
          const uint32_t q_a = smem_u32(base + kOffQ + qb * kTileBytes);
          const uint32_t g_a = smem_u32(base + kOffG + qb * kGSetBytes);   // K_G, Q_G, V_G
          uint32_t committed = 0;
          if (pg_pending &&
              !(ok = mbar_wait(&sm.bar_pvdone[kNoSlot], (item_no - 1) & 1, abort_flag)))
            break;
          pg_pending = false;
          if (!(ok = mbar_wait(&sm.bar_q[qb], (item_no >> 1) & 1, abort_flag))) break;
          tc_fence_after();
          auto s_free = [&]() -> bool {
            return s_uses == 0 || mbar_wait(&sm.bar_sfree, (s_uses - 1) & 1, abort_flag);
          };
          auto issue_pv = [&](int t) -> bool {
            if (!mbar_wait(&sm.bar_pready[n_p & 1], (n_p >> 1) & 1, abort_flag)) return false;
            ++n_p;
            const int vs = vc % kBandVStages;
            if (!mbar_wait(&sm.bar_vfull[vs], (vc / kBandVStages) & 1, abort_flag)) return false;
            // the first product overwrites O: the helpers have read the previous item's
            if (t == 0 && item_no > 0 && !mbar_wait(&sm.bar_ofree, (item_no - 1) & 1, abort_flag))
              return false;
            tc_fence_after();
            mma_pv_ts(tm + kColO, tm + col_slot(t), v_a + vs * kTileBytes, kTile / 16, t > 0);
            umma_commit(&sm.bar_vempty[vs]);
            umma_commit(&sm.bar_pvdone[t]);
            committed |= 1u << t;
            ++vc;
            return true;
          };
          for (int t = 0; ok && t < x.nk; ++t) {
            const int ks = kc % kBandKStages;
            if (!(ok = s_free())) break;
            if (!(ok = mbar_wait(&sm.bar_kfull[ks], (kc / kBandKStages) & 1, abort_flag))) break;
            tc_fence_after();
            mma_qk(tm + kColS, q_a, k_a + ks * kTileBytes, 128);   // S_t
            umma_commit(&sm.bar_sfull);
            ++s_uses;
            if (t == x.diag && glob) {   // S_Gt: this key tile against the global queries
              if (!(ok = s_free())) break;
              tc_fence_after();
              mma_qk(tm + kColS, k_a + ks * kTileBytes, g_a + kGTileBytes, 16);
              umma_commit(&sm.bar_sfull);
              ++s_uses;
            }
            umma_commit(&sm.bar_kempty[ks]);
            ++kc;
            if (t > 0 && !(ok = issue_pv(t - 1))) break;
          }
          if (ok) ok = issue_pv(x.nk - 1);
          if (ok && glob) {   // S_G = Q K_G^T, then P_G V_G
            if ((ok = s_free())) {
              tc_fence_after();
              mma_qk(tm + kColS, q_a, g_a, 16);
              umma_commit(&sm.bar_sfull);
              ++s_uses;
              ok = mbar_wait(&sm.bar_pgready, n_glob & 1, abort_flag);
              ++n_glob;
            }
            if (ok) {
              tc_fence_after();
              mma_pv_ts(tm + kColO, tm + kColPG, g_a + 2 * kGTileBytes, kMaxGlobal / 16, true);
              umma_commit(&sm.bar_pvdone[kNoSlot]);
              committed |= 1u << kNoSlot;
              pg_pending = true;
            }
          }
          if (!ok) break;
          // every P V barrier completes one phase per item
          for (int u = 0; u <= kMaxBandTiles; ++u)
            if (!((committed >> u) & 1u)) umma_commit(&sm.bar_pvdone[u]);
          umma_commit(&sm.bar_qfree[qb]);
          ++item_no;
        }
        umma_commit(&sm.bar_fin);
        drain_wait(&sm.bar_fin, 0);
      }
      __syncwarp();
    } else {
      // ------------------------------------------- column-sum products
      if (lane == 0) {
        const uint32_t st_a = smem_u32(base + kOffStage);
        uint32_t item_no = 0, st_n = 0;
        bool ok = true;
        for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x) {
          const BandItem x = band_item(p, v, it);
          if (!x.run) continue;
          if (!(ok = mbar_wait(&sm.bar_epi, item_no & 1, abort_flag))) break;
          const uint32_t w_a = smem_u32(base + kOffW + (item_no & 1) * kWBytes);
          for (int t = 0; ok && t < x.nk; ++t) {
            const int u = st_n & 1;
            if (!(ok = mbar_wait(&sm.bar_stfull[u], (st_n >> 1) & 1, abort_flag))) break;
            ++st_n;
            tc_fence_after();
            mma_colsum(tm + col_slot(t), st_a + u * kStageBytes, w_a);
            umma_commit(&sm.bar_stfree[u]);
            umma_commit(&sm.bar_dfull[t]);
          }
          if (!ok) break;
          for (int t = x.nk; t < kMaxBandTiles; ++t) umma_commit(&sm.bar_dfull[t]);
          ++item_no;
        }
        umma_commit(&sm.bar_fin2);
        drain_wait(&sm.bar_fin2, 0);
      }
      __syncwarp();
    }
  } else if (warp >= 8) {
    // --------------------------------------------------------- helpers: the
    // epilogue of each item, while the softmax warps run the next one
    regs_dealloc<kBandHelperRegs>();
    const int q4 = warp & 3, r = 32 * q4 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
    uint8_t* stage = base + kOffStage;
    uint32_t item_no = 0, st_n = 0;
    bool ok = true;
    for (int it = blockIdx.x; it < n_items; it += gridDim.x) {
      const BandItem x = band_item(p, v, it);
      if (!x.run) continue;
      ok = ok && warp_wait(&sm.bar_epi, item_no & 1, abort_flag);
      // O = (sum of the P~ V products) / osum, through this warp's rows of staging buffer 1
      const float inv = sm.inv_osum[item_no & 1][r];
      if (ok && v.O != nullptr) {
        tc_fence_after();
        uint8_t* ost = stage + kStageBytes + q4 * 8192;
#pragma unroll
        for (int c = 0; c < 64; c += 32) {
          float o[32];
          tmem_ld32(tm + kColO + c + lane_off, o);
          tmem_ld_wait();
#pragma unroll
          for (int k = 0; k < 32; k += 8)
            stage_row_piece<8>(ost, (c + k) >> 3,
                               make_uint4(pack_bf16x2(o[k] * inv, o[k + 1] * inv),
                                          pack_bf16x2(o[k + 2] * inv, o[k + 3] * inv),
                                          pack_bf16x2(o[k + 4] * inv, o[k + 5] * inv),
                                          pack_bf16x2(o[k + 6] * inv, o[k + 7] * inv)));
        }
        flush_staged_rows<8>(
            ost, v.O + ((static_cast<size_t>(x.b) * p.L + x.q * kTile + 32 * q4) * p.H + x.h) * kHeadDim,
            static_cast<size_t>(p.H) * kHeadDim, __ballot_sync(0xffffffffu, inv > 0.f));
      }
      tc_fence_before();
      warp_arrive(&sm.bar_ofree);

      // the column sums: D_t[key][2t] + D_t[key][2t + 1], one per key of band tile t;
      // slot t goes back to the softmax warps once read
      auto read_d = [&](int t) {
        const bool ok3 = ok && (ok = warp_wait(&sm.bar_dfull[t], item_no & 1, abort_flag));
        const int j = (x.klo + t) * kTile + r;
        if (ok3) {
          tc_fence_after();
          float d0, d1;
          tmem_ld2(tm + col_slot(t) + 2 * t + lane_off, d0, d1);
          tmem_ld_wait();
          if (j < x.n)
            p.colpart[((static_cast<size_t>(x.b) * p.H + x.h) * p.L + j) * p.band_slots +
                      x.q % p.band_slots] = d0 + d1;
        }
        tc_fence_before();
        warp_arrive(&sm.bar_slotfree[t]);
      };
      // stage each tile's P~ transposed for its column-sum product (two buffers)
      for (int t = 0; t < x.nk; ++t) {
        const int u = st_n & 1;
        if (ok && st_n >= 2) ok = warp_wait(&sm.bar_stfree[u], ((st_n >> 1) - 1) & 1, abort_flag);
        ++st_n;
        if (ok) {
          tc_fence_after();
          uint32_t w[64];
          tmem_ld32(tm + col_slot(t) + lane_off, reinterpret_cast<float*>(w));
          tmem_ld32(tm + col_slot(t) + 32 + lane_off, reinterpret_cast<float*>(w + 32));
          tmem_ld_wait();
          uint8_t* st = stage + u * kStageBytes;
#pragma unroll
          for (int a = 0; a < 2; ++a)
#pragma unroll
            for (int c = 0; c < 8; ++c)
              *reinterpret_cast<uint4*>(st + stage_offset_mn(r, a, c)) =
                  make_uint4(w[32 * a + 4 * c], w[32 * a + 4 * c + 1], w[32 * a + 4 * c + 2],
                             w[32 * a + 4 * c + 3]);
          fence_proxy_async_smem();
        }
        tc_fence_before();
        warp_arrive(&sm.bar_stfull[u]);
        if (t > 0) read_d(t - 1);
      }
      read_d(x.nk - 1);
      for (int t = x.nk; t < kMaxBandTiles; ++t) warp_arrive(&sm.bar_slotfree[t]);
      // the item's results (O, column sums, and the softmax warps' global-token
      // pieces written before bar_epi) are visible to the cols CTAs
      if (helpers_sync_or(!ok)) {
        ok = false;
        break;
      }
      if (r == 0) {
        __threadfence();
        red_release_add_u32(p.rows_done + x.b * p.H + x.h, 1u);
      }
      ++item_no;
    }
  } else {
    // --------------------------------------------------------- softmax
    regs_alloc<kBandSoftmaxRegs>();
    const int q4 = warp & 3, hf = warp >> 2, r = 32 * q4 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(q4 * 32) << 16;
    uint32_t n_sfull = 0, n_p = 0, item_no = 0, n_pair = 0;
    bool ok = true;
    // the partner warp's value of row r, exchanged through shared memory
    auto pair_max = [&](float mine) -> float {
      sm.xmax[n_pair & 1][hf][r] = mine;
      warp_arrive(&sm.bar_pair[q4]);
      const bool w_ok = warp_wait(&sm.bar_pair[q4], n_pair & 1, abort_flag);
      const float other = sm.xmax[n_pair & 1][hf ^ 1][r];
      ++n_pair;
      ok = ok && w_ok;
      return fmaxf(mine, other);
    };
    for (int it = blockIdx.x; ok && it < n_items; it += gridDim.x) {
      const BandItem x = band_item(p, v, it);
      if (!x.run) continue;
      const bool glob = x.ng > 0;
      // lane g < ng holds the current index of global token g
      const int my_gc = lane < x.ng ? __ldcg(v.gcur + x.b * kMaxGlobal + lane) : -1;
      const int i = x.q * kTile + r;   // current index of this query row
      bool row_global = false;
      for (int g = 0; g < x.ng; ++g) row_global |= (__shfl_sync(0xffffffffu, my_gc, g) == i);
      const bool valid = (i < x.n) && !row_global;
      // allowed band keys of this row, inclusive; rows whose results are not
      // kept (global rows, rows past the end) take no key: their P~ is zero
      const int lo = valid ? max(0, i - p.w) : x.n;
      const int hi = valid ? min(x.n - 1, i + p.w) : -1;

      float m_ref = -INFINITY, lsum = 0.f, osum = 0.f;
      float m0 = -INFINITY, m1 = -INFINITY, m2 = -INFINITY, m3 = -INFINITY, m4 = -INFINITY;
      uint32_t pv_sent = 0;   // P V products of this item handed to the MMA thread (bit t)

      // Running reference m_ref (base 2): P~ = exp2(x - m_ref), raised when a
      // tile's maximum exceeds it by more than 8; O and both row sums are then
      // rescaled exactly (after every P V handed over so far has completed).
      // Each tile's P~ keeps the reference it was taken with (m0..m4) for the
      // column sums.
      auto raise_to = [&](float tmax) -> bool {
        const bool raise = tmax > m_ref + 8.f;
        float f = 1.f;
        if (raise) {
          f = (m_ref == -INFINITY) ? 0.f : ex2(m_ref - tmax);
          m_ref = tmax;
          lsum *= f;
          osum *= f;
        }
        if (__any_sync(0xffffffffu, raise) && pv_sent != 0) {
          const int last = pv_sent >> kNoSlot ? kNoSlot : 31 - __clz(pv_sent);
          if (!warp_wait(&sm.bar_pvdone[last], item_no & 1, abort_flag)) return false;
          tc_fence_after();
          rescale_o(tm + kColO + 32 * hf + lane_off, f);
        }
        return true;
      };

      for (int t = 0; ok && t < x.nk; ++t) {
        const int j0 = (x.klo + t) * kTile + 64 * hf;
        const int a = lo - j0, e = hi - j0;   // allowed keys of this half: a .. e
        if (!(ok = warp_wait(&sm.bar_sfull, (n_sfull++) & 1, abort_flag))) break;
        tc_fence_after();
        float xs[64];
        tmem_ld32(tm + kColS + 64 * hf + lane_off, xs);
        tmem_ld32(tm + kColS + 64 * hf + 32 + lane_off, xs + 32);
        tmem_ld_wait();
        tc_fence_before();
        warp_arrive(&sm.bar_sfree);   // S is in registers: the next product may overwrite it
        if (t == x.diag && glob) {
          // S_Gt follows in the S columns
          if (!(ok = warp_wait(&sm.bar_sfull, (n_sfull++) & 1, abort_flag))) break;
          if (hf == 0) {
            float xt[kMaxGlobal];
            tc_fence_after();
            tmem_ld16(tm + kColS + lane_off, xt);
            tmem_ld_wait();
            tc_fence_before();
            warp_arrive(&sm.bar_sfree);
            global_query_stats(p, x, q4, r, xt);
          } else {
            tc_fence_before();
            warp_arrive(&sm.bar_sfree);
          }
        }
        bool alive0 = true, alive1 = true;
        if (!__all_sync(0xffffffffu, a <= 0 && e >= 63)) {
#pragma unroll
          for (int ch = 0; ch < 2; ++ch) {
            const uint32_t keep = bit_range32(a - 32 * ch, e - 32 * ch);
            if (!__any_sync(0xffffffffu, keep != 0u)) {
              if (ch == 0) alive0 = false;
              else alive1 = false;
#pragma unroll
              for (int k = 0; k < 32; ++k) xs[32 * ch + k] = -INFINITY;
            } else if (__any_sync(0xffffffffu, keep != 0xffffffffu)) {
#pragma unroll
              for (int k = 0; k < 32; ++k) {
                const uint32_t out =
                    ~static_cast<uint32_t>(static_cast<int32_t>(keep << (31 - k)) >> 31);
                xs[32 * ch + k] = __uint_as_float((__float_as_uint(xs[32 * ch + k]) & ~out) |
                                                  (0xff800000u & out));
              }
            }
          }
        }
        float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
        for (int k = 0; k < 64; k += 8) {
          mx4[0] = fmax3(mx4[0], xs[k], xs[k + 1]);
          mx4[1] = fmax3(mx4[1], xs[k + 2], xs[k + 3]);
          mx4[2] = fmax3(mx4[2], xs[k + 4], xs[k + 5]);
          mx4[3] = fmax3(mx4[3], xs[k + 6], xs[k + 7]);
        }
        const float tmax =
            pair_max(fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3])) * kLogitScale2);
        if (!ok) break;
        if (!(ok = raise_to(tmax))) break;
        // the slot is free once the previous item's column sums of it have been read
        if (item_no > 0 && !(ok = warp_wait(&sm.bar_slotfree[t], (item_no - 1) & 1, abort_flag)))
          break;
        exp_half_tile(xs, m_ref == -INFINITY ? 0.f : -m_ref, alive0, alive1,
                      tm + col_slot(t) + 32 * hf + lane_off, lsum, osum);
        if (t == 0) m0 = m_ref;
        else if (t == 1) m1 = m_ref;
        else if (t == 2) m2 = m_ref;
        else if (t == 3) m3 = m_ref;
        else m4 = m_ref;
        tmem_st_wait();
        tc_fence_before();
        warp_arrive(&sm.bar_pready[(n_p++) & 1]);
        pv_sent |= 1u << t;
      }

      // ---- the global keys outside the row's band: one more block of the softmax
      float pgf[kMaxGlobal];
#pragma unroll
      for (int g = 0; g < kMaxGlobal; ++g) pgf[g] = 0.f;
      if (ok && glob) {
        if ((ok = warp_wait(&sm.bar_sfull, (n_sfull++) & 1, abort_flag))) {
          float xg[kMaxGlobal];
          float gmax = -INFINITY;
          if (hf == 0) {
            tc_fence_after();
            tmem_ld16(tm + kColS + lane_off, xg);
            tmem_ld_wait();
#pragma unroll
            for (int g = 0; g < kMaxGlobal; ++g) {
              const int gc = __shfl_sync(0xffffffffu, my_gc, g);
              const bool use = valid && g < x.ng && abs(i - gc) > p.w;
              xg[g] = use ? xg[g] * kLogitScale2 : -INFINITY;
              gmax = fmaxf(gmax, xg[g]);
            }
          }
          tc_fence_before();
          warp_arrive(&sm.bar_sfree);
          const float tmax = pair_max(gmax);
          if (ok) ok = raise_to(tmax);
          if (ok && hf == 0) {
            const float nref = (m_ref == -INFINITY) ? 0.f : -m_ref;
            uint32_t pg[kMaxGlobal / 2];
#pragma unroll
            for (int g = 0; g < kMaxGlobal; g += 2) {
              pgf[g] = ex2(xg[g] + nref);
              pgf[g + 1] = ex2(xg[g + 1] + nref);
              pg[g / 2] = pack_bf16x2(pgf[g], pgf[g + 1]);
              lsum += pgf[g] + pgf[g + 1];
              osum = add_bf16_hi(add_bf16_lo(osum, pg[g / 2]), pg[g / 2]);
            }
            tmem_st8(tm + kColPG + lane_off, pg);
            tmem_st_wait();
            tc_fence_before();
            warp_arrive(&sm.bar_pgready);
          }
        }
      }

      // ---- epilogue: every P V of the item complete, the row totals of both
      // halves, LSE, the weights of the column sums, the global keys' far-row sums
      const int lastpv = glob ? kNoSlot : x.nk - 1;
      const bool have = ok && warp_wait(&sm.bar_pvdone[lastpv], item_no & 1, abort_flag);
      ok = have;
      sm.xsum[item_no & 1][hf][0][r] = lsum;
      sm.xsum[item_no & 1][hf][1][r] = osum;
      warp_arrive(&sm.bar_pair[q4]);
      ok = warp_wait(&sm.bar_pair[q4], n_pair & 1, abort_flag) && ok;
      ++n_pair;
      const float lsum_t = lsum + sm.xsum[item_no & 1][hf ^ 1][0][r];
      const float osum_t = osum + sm.xsum[item_no & 1][hf ^ 1][1][r];
      const float lse = (ok && valid) ? m_ref + lg2(lsum_t) : INFINITY;
      // W[2t][i] + W[2t + 1][i] = c_{i,t} = 2^(m_t - LSE_i), split into two bf16
      uint8_t* W = base + kOffW + (item_no & 1) * kWBytes;
#pragma unroll
      for (int t = 0; t < kMaxBandTiles; ++t) {
        if (t >= x.nk) break;
        if ((t & 1) != hf) continue;
        const float mt = t == 0 ? m0 : t == 1 ? m1 : t == 2 ? m2 : t == 3 ? m3 : m4;
        const float c = (lse == INFINITY || mt == -INFINITY) ? 0.f : ex2(mt - lse);
        const __nv_bfloat16 chi = __float2bfloat16_rn(c);
        const __nv_bfloat16 clo = __float2bfloat16_rn(c - __bfloat162float(chi));
        *reinterpret_cast<__nv_bfloat16*>(W + w_offset(2 * t, r)) = chi;
        *reinterpret_cast<__nv_bfloat16*>(W + w_offset(2 * t + 1, r)) = clo;
      }
      if (hf == 0) sm.inv_osum[item_no & 1][r] = (ok && valid) ? 1.f / osum_t : 0.f;
      if (glob && hf == 0) {
        // far-row column sums of the global keys, per 32-row warp slice
        const size_t slot0 =
            (((static_cast<size_t>(x.b) * p.H + x.h) * p.T + x.q) * 4 + q4) * kMaxGlobal;
        const float cg = (lse == INFINITY) ? 0.f : ex2(m_ref - lse);
#pragma unroll
        for (int g = 0; g < kMaxGlobal; ++g) pgf[g] *= cg;
        const float gsum = warp_reduce16(pgf, OpAdd());
        const int gme = lane >> 1;
        if ((lane & 1) == 0 && gme < x.ng) p.gpart[slot0 + gme] = gsum;
      }
      fence_proxy_async_smem();   // W is read by the tensor cores
      tc_fence_before();
      warp_arrive(&sm.bar_epi);
      ++item_no;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 15) {
    tc_fence_after();
    tmem_dealloc(tm, 512);
  }
  if (tid == 0 && sm.abort) atomicOr(p.status, kStatusTimeout);
}

cudaError_t configure_band() {
  // the warpgroups' register split (setmaxnreg) needs the whole launch
  // allocation: with fewer registers a thread, an increase would never be granted
  cudaFuncAttributes fa;
  cudaError_t e = cudaFuncGetAttributes(&fa, sc_band_kernel);
  if (e == cudaSuccess && fa.numRegs * kBandThreads < 65536) e = cudaErrorInvalidConfiguration;
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(sc_band_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(kBandDyn));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(sc_band_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
  return e;
}

cudaError_t launch_band(const TensorMaps& m, const LayerParams& p, int sms, cudaStream_t st) {
  const int items = p.B * p.H * p.T;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(items < sms ? items : sms));
  cfg.blockDim = dim3(kBandThreads);
  cfg.dynamicSmemBytes = kBandDyn;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, sc_band_kernel, m, p);
}

}  // namespace sc
