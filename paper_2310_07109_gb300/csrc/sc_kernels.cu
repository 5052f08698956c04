// sc_kernels.cu -- device code of one sparse-attention + learned-token-pruning
// layer on sm_103a.
//
// Per layer, per sequence b (n current tokens, original positions pos[b][*]):
//
//   rows kernel   (one CTA per pair of 128-row query tiles of one (sequence,
//                 head); one softmax warpgroup per tile)
//     S = Q K^T over the band key tiles and one 16-wide tile of global keys on
//     the tensor cores (tcgen05, bf16 -> fp32 in tensor memory); each 16 KB
//     operand tile is one TMA copy.  Row softmax in fp32 (base 2, lazily
//     rescaled running max); P (bf16) goes back to tensor memory and P V
//     accumulates there.  Then the band pass: S^T = K Q^T of each key tile of
//     the band (the tiles are still resident) and, per key column j, the sum
//     over the tile's rows of exp2(S_ij - LSE_i) (one thread per column, no
//     cross-thread reduction), one partial per (key, query tile).  Writes O,
//     the row log-sum-exp LSE_i, those partials, the far-row column sums of
//     the global keys, and (max, sum) of the global rows over this tile's keys.
//
//   cols kernel   (one CTA per pair of 128-key tiles; one warpgroup per tile)
//     The global rows' probabilities over the pair's keys and their P V
//     outputs, and each key's column sum: the band partials added in tile
//     order, plus the global rows' share.  The last CTA of a key-tile pair
//     sums the heads in a fixed order and applies the threshold; the last pair
//     of a sequence compacts the survivors in order.  Each CTA waits (bounded)
//     only for the rows CTAs of its own (sequence, head); the "last" CTAs are
//     found by atomic counters.
//
//   gather kernel copies the survivors' next-layer Q, K, V rows into compacted
//   buffers (coalesced 16-byte vectors) when they are not already in place.
//
// The method (allowed sets, row softmax, vertical accumulation, >= threshold,
// order-preserving removal) is Sec. "Sparse Attention", Sec. "Extractor of
// Attention Scores in Sparse Attention Matrix" and Sec. "Token Pruning".
#include <algorithm>
#include <cuda_runtime.h>
#include <utility>
#include <cuda_bf16.h>
#include <cstdint>

#include "sc_internal.cuh"
#include "sc_layer_common.cuh"
#include "sc_select.cuh"
#include "sm103_primitives.cuh"

namespace sc {

// ---------------------------------------------------------------------------
// rows kernel
// ---------------------------------------------------------------------------
// One CTA per pair of 128-row query tiles (2p, 2p+1) of one (sequence, head),
// one softmax warpgroup per tile; the two tiles share their K/V tiles (the
// band of the pair spans at most six 128-key tiles: all K tiles stay
// resident, V tiles pass through a ring) and one tensor core serves both.
//
// Per key tile a warpgroup loads all 128 columns of S into registers and
// hands that tensor memory straight back, so S of its next key tile is
// computed while it evaluates this tile's exponentials.  P (bf16) goes to its
// own tensor-memory columns and P V reads it from there (no shared-memory
// traffic for P).
//
// Tensor memory (512 columns) per warpgroup X in {0, 1}, base 256 X:
//   S    [+0, +128)   S of the current key tile (fp32); after the last tile:
//                     S_G [+0, +16) (the 16 global keys) and S_Gt [+16, +32)
//                     (the diagonal key tile against the global queries)
//   P    [+128, +192) P of the current key tile, bf16 pairs; before the
//                     first tile: S_G [+128, +144) and P_G [+144, +152)
//   O    [+192, +256)
// Warps 0-7: the two softmax warpgroups; warpgroup 2 (warps 8-11): warp 8
// loads Q and the K tiles, warp 10 the V tiles, warps 9 and 11 issue the MMAs
// of softmax warpgroups 0 and 1 (one issuing thread per warpgroup, so each
// tcgen05.commit covers that warpgroup's MMAs only).
// Launched at 168 registers a thread (three warps per SM sub-partition);
// warpgroup 2 gives registers back so that the softmax warps, which hold a
// whole 128-column row of S, get 200: 128 x 96 + 256 x 200 = 63488 <= 384 x 168.
constexpr int kRowsThreads = 384;
constexpr int kRowsLaunchRegs = 168;
constexpr int kRowsCtlRegs = 96;
constexpr int kRowsSoftmaxRegs = 200;
static_assert(128 * kRowsCtlRegs + 256 * kRowsSoftmaxRegs <= kRowsThreads * kRowsLaunchRegs,
              "register split exceeds the launch allocation");
constexpr int kPairTiles = kMaxBandTiles + 1;
// V slots: with six key tiles only the sixth reuses a slot, that of the first;
// the first is used by query tile 0 alone and the sixth by query tile 1 alone
// (each query tile's band spans at most five key tiles).
constexpr int kVStages = kPairTiles - 1;
// Wide windows (256 < w <= 512 on sequences of more than five tiles): one
// query tile per CTA, up to nine resident key tiles and a three-slot V ring in
// the same shared memory (one Q tile + 9 + 3 = two Q tiles + 6 + 5).
constexpr int kWideVStages = 3;
static_assert(1 + kWideBandTiles + kWideVStages == 2 + kPairTiles + kVStages,
              "both layouts fill the same shared memory");

__host__ __device__ constexpr uint32_t col_s(int X) { return 256u * X; }
__host__ __device__ constexpr uint32_t col_p(int X) { return 256u * X + 128u; }
__host__ __device__ constexpr uint32_t col_o(int X) { return 256u * X + 192u; }

struct RowsSmem {
  alignas(16) float nlse[2][kTile];   // -LSE of each query tile's rows (read as float4)
  uint64_t bar_q;
  uint64_t bar_kfull[kWideBandTiles];
  uint64_t bar_vfull[kVStages], bar_vempty[kVStages];
  uint64_t bar_sg[2], bar_sgend[2], bar_sfull[2], bar_sfree[2], bar_pready[2], bar_pvdone[2];
  uint64_t bar_fin[2];
  uint64_t bar_stall;   // test hook: nothing ever completes it
  uint32_t tmem_base;
  int abort;
  int gc[kMaxGlobal];
};

// dynamic shared memory: two Q tiles, every K tile of the pair, the V ring,
// the global rows
constexpr uint32_t kRowsDyn =
    kTileBytes * (2 + kPairTiles + kVStages) + 3 * kGTileBytes + 1024;

// kWide: one query tile per CTA (see kWideVStages); otherwise pairs of tiles.
template <bool kWide>
__global__ void __launch_bounds__(kRowsThreads, 1)
    sc_rows_kernel(const __grid_constant__ TensorMaps maps, const __grid_constant__ LayerParams p) {
  // the cols kernel is scheduled once every CTA here has passed this wait, so
  // what the kernels before this one wrote is complete when it starts (with
  // p.gathered, the gather kernel before this one lets it start only once the
  // kernels before the gather are complete, and each CTA waits below for its
  // own sequence's rows)
  if (p.gathered == nullptr) pdl_wait();
  pdl_launch_dependents();
  // grid: pairs of query tiles (single tiles with a wide window),
  // (sequence, head)-major, so that the CTAs of a (sequence, head) finish
  // together and its cols CTAs can start early
  constexpr bool wide = kWide;
  constexpr int band_slots = wide ? kWideBandTiles : kMaxBandTiles;
  const int per_bh = wide ? p.T : (p.T + 1) / 2;
  const int pr = blockIdx.x % per_bh, bh = blockIdx.x / per_bh;
  const int h = bh % p.H, b = bh / p.H;
  const int q_first = wide ? pr : 2 * pr;   // first query tile of this CTA
  const LayerView v = layer_view(p);
  // the sequence's state, loaded together
  const bool tailed = owned_by_tail(p, v, b);
  const int n = __ldcg(v.len + b);
  const int ng_raw = __ldcg(v.ng + b);
  const int gc_raw = threadIdx.x < kMaxGlobal ? __ldcg(v.gcur + b * kMaxGlobal + threadIdx.x) : -1;
  if (tailed) return;
  if (q_first * kTile >= n) return;
  const int ng = min(ng_raw, kMaxGlobal);
  const int ngp = ng > 0 ? kMaxGlobal : 0;
  const bool hasB = !wide && (q_first + 1) * kTile < n;
  constexpr int nvs = wide ? kWideVStages : kVStages;   // V ring slots

  extern __shared__ uint8_t dyn_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dyn_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* Qs = base;                                        // 2 tiles (wide: 1)
  uint8_t* Ks = Qs + (wide ? 1 : 2) * kTileBytes;            // all resident: 6 (wide: 9)
  uint8_t* Vs = Ks + (wide ? kWideBandTiles : kPairTiles) * kTileBytes;   // nvs slots
  uint8_t* KG = Vs + nvs * kTileBytes;
  uint8_t* VG = KG + kGTileBytes;
  uint8_t* QG = VG + kGTileBytes;
  __shared__ RowsSmem sm;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // key tiles of each query tile, and of the pair (absolute tile indices)
  int klo[2], khi[2];
#pragma unroll
  for (int X = 0; X < 2; ++X) {
    const int q0 = (q_first + X) * kTile, q1 = min(q0 + kTile - 1, n - 1);
    klo[X] = max(0, q0 - p.w) / kTile;
    khi[X] = min(n - 1, q1 + p.w) / kTile;
  }
  const int kt_lo = klo[0];
  const int kt_hi = hasB ? khi[1] : khi[0];
  const int nk = kt_hi - kt_lo + 1;   // <= 6 (wide: 9); window checked on the host

  if (tid == 0) {
    mbar_init(&sm.bar_q, 1);
    for (int k = 0; k < kWideBandTiles; ++k) mbar_init(&sm.bar_kfull[k], 1);
    for (int s = 0; s < kVStages; ++s) {
      mbar_init(&sm.bar_vfull[s], 1);
      mbar_init(&sm.bar_vempty[s], 1);
    }
    for (int X = 0; X < 2; ++X) {
      mbar_init(&sm.bar_sg[X], 1);
      mbar_init(&sm.bar_sgend[X], 1);
      mbar_init(&sm.bar_sfull[X], 1);
      mbar_init(&sm.bar_sfree[X], 4);   // one arrival per warp
      mbar_init(&sm.bar_pready[X], 4);
      mbar_init(&sm.bar_pvdone[X], 1);
      mbar_init(&sm.bar_fin[X], 1);
    }
    mbar_init(&sm.bar_stall, 1);
    sm.abort = 0;
    fence_mbar_init();
    // this sequence's rows may still be crossing the host link
    if (p.gathered != nullptr) wait_count(p.gathered + b, p.gather_target, &sm.abort);
  }
  if (tid < kMaxGlobal) sm.gc[tid] = tid < ng ? gc_raw : -1;
  if (warp == 9) tmem_alloc(&sm.tmem_base, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (p.gathered != nullptr) fence_proxy_async_global();   // the copies, before any TMA load
  const uint32_t tm = sm.tmem_base;
  volatile int* abort_flag = &sm.abort;

  if (warp >= 8) {
   regs_dealloc<kRowsCtlRegs>();
   if (warp == 8) {
    // ------------------------------------------------------------- Q, globals, K
    const RowSource rs = row_source(p, v, b);
    if (lane == 0) {
      // Q, then the first two K tiles (the first S needs Q and K), then the
      // global rows, then the other K tiles
      mbar_arrive_expect_tx(&sm.bar_q, (hasB ? 2 : 1) * kTileBytes + 3 * ngp * 128);
      load_tile(maps, 0, rs, h, q_first * kTile, Qs, &sm.bar_q);
      if (hasB) load_tile(maps, 0, rs, h, (q_first + 1) * kTile, Qs + kTileBytes, &sm.bar_q);
      for (int k = 0; k < nk && k < 2; ++k) {
        mbar_arrive_expect_tx(&sm.bar_kfull[k], kTileBytes);
        load_tile(maps, 1, rs, h, (kt_lo + k) * kTile, Ks + k * kTileBytes, &sm.bar_kfull[k]);
      }
    }
    __syncwarp();
    if (ngp) {
      load_globals(maps, 1, rs, h, p.H, sm.gc, ng, KG, &sm.bar_q, lane);
      load_globals(maps, 2, rs, h, p.H, sm.gc, ng, VG, &sm.bar_q, lane);
      load_globals(maps, 0, rs, h, p.H, sm.gc, ng, QG, &sm.bar_q, lane);
    }
    if (lane == 0) {
      for (int k = 2; k < nk; ++k) {
        mbar_arrive_expect_tx(&sm.bar_kfull[k], kTileBytes);
        load_tile(maps, 1, rs, h, (kt_lo + k) * kTile, Ks + k * kTileBytes, &sm.bar_kfull[k]);
      }
      // nothing may still be landing in shared memory when the CTA exits
      drain_wait(&sm.bar_q, 0);
      for (int k = 0; k < nk; ++k) drain_wait(&sm.bar_kfull[k], 0);
    }
   } else if (warp == 10) {
    // ------------------------------------------------------------- V ring
    if (lane == 0) {
      const RowSource rs = row_source(p, v, b);
      bool ok = true;
      int issued = 0;
      // slot s = k mod nvs and its use count, advanced without division
      for (int k = 0, s = 0, use = 0; ok && k < nk; ++k) {
        if (k >= nvs && !(ok = mbar_wait(&sm.bar_vempty[s], (use - 1) & 1, abort_flag))) break;
        mbar_arrive_expect_tx(&sm.bar_vfull[s], kTileBytes);
        load_tile(maps, 2, rs, h, (kt_lo + k) * kTile, Vs + s * kTileBytes, &sm.bar_vfull[s]);
        issued = k + 1;
        if (++s == nvs) {
          s = 0;
          ++use;
        }
      }
      // the last copy issued into each slot has landed (after an expired wait
      // fewer than nk were issued)
      for (int s = 0; s < nvs && s < issued; ++s) {
        const int last = s + nvs * ((issued - 1 - s) / nvs);
        drain_wait(&sm.bar_vfull[s], (last / nvs) & 1);
      }
    }
   } else if (warp == 9 || warp == 11) {
    // ------------------------------------------------------------- MMA issue
    const int X = warp == 9 ? 0 : 1;
    if (lane == 0 && (X == 0 || hasB)) {
      const uint32_t q_a = smem_u32(Qs) + X * kTileBytes, k_a = smem_u32(Ks), v_a = smem_u32(Vs);
      const int kloX = klo[X], khiX = khi[X];
      const uint32_t tS = tm + col_s(X), tP = tm + col_p(X), tO = tm + col_o(X);
      bool ok = true;
      if (X == 0 && p.stall_ns != 0)   // test hook: this bounded wait expires
        ok = mbar_wait(&sm.bar_stall, 0, abort_flag, p.stall_ns);
      ok = ok && mbar_wait(&sm.bar_q, 0, abort_flag);
      if (ok) {
        tc_fence_after();
        if (ngp) {
          mma_qk(tP, q_a, smem_u32(KG), 16);   // S_G
          umma_commit(&sm.bar_sg[X]);
        }
      }
      // This warpgroup's events come in a fixed order: [P_G stored], then per
      // key tile "S read" (sfree) and "P stored" (pready).  S of the next
      // tile is issued at "S read", P V of a tile at "P stored".
      auto issue_s = [&](int a) -> bool {
        const int k = a - kt_lo;
        if (!mbar_wait(&sm.bar_kfull[k], 0, abort_flag)) return false;
        tc_fence_after();
        mma_qk(tS, q_a, k_a + k * kTileBytes, 128);
        umma_commit(&sm.bar_sfull[X]);
        return true;
      };
      uint32_t nfree = 0, nready = 0;
      // V slot of key tile k = a - kt_lo (k mod nvs) and its use count, advanced
      // without division
      int vslot = (kloX - kt_lo) % nvs, vuse = (kloX - kt_lo) / nvs;
      if (ok) ok = issue_s(kloX);
      if (ok && ngp) {
        if ((ok = mbar_wait(&sm.bar_pready[X], (nready++) & 1, abort_flag))) {
          tc_fence_after();
          mma_pv_ts(tO, tP + 16, smem_u32(VG), kMaxGlobal / 16, false);   // P_G V_G
          umma_commit(&sm.bar_pvdone[X]);
        }
      }
      for (int a = kloX; ok && a <= khiX; ++a) {
        const int k = a - kt_lo;
        if (!(ok = mbar_wait(&sm.bar_sfree[X], (nfree++) & 1, abort_flag))) break;
        if (a < khiX) {
          if (!(ok = issue_s(a + 1))) break;
        } else if (ngp) {
          // the last S is read: its columns take S_G and S_Gt for the epilogue
          tc_fence_after();
          mma_qk(tS, q_a, smem_u32(KG), 16);
          mma_qk(tS + 16, k_a + (q_first + X - kt_lo) * kTileBytes, smem_u32(QG), 16);
          umma_commit(&sm.bar_sgend[X]);
        }
        if (!(ok = mbar_wait(&sm.bar_pready[X], (nready++) & 1, abort_flag))) break;
        if (!(ok = mbar_wait(&sm.bar_vfull[vslot], vuse & 1, abort_flag))) break;
        tc_fence_after();
        mma_pv_ts(tO, tP, v_a + vslot * kTileBytes, kTile / 16, ngp > 0 || a > kloX);
        if (k + nvs < nk) umma_commit(&sm.bar_vempty[vslot]);   // slot reused
        if (++vslot == nvs) {
          vslot = 0;
          ++vuse;
        }
        umma_commit(&sm.bar_pvdone[X]);
      }
      // band pass: S^T = K Q^T of each key tile of the band against this
      // query tile, into the S columns once they are read (after the S_G /
      // S_Gt of the epilogue, when there are global keys)
      for (int a = kloX; ok && a <= khiX; ++a) {
        if ((a > kloX || ngp) && !(ok = mbar_wait(&sm.bar_sfree[X], (nfree++) & 1, abort_flag)))
          break;
        tc_fence_after();
        mma_qk(tS, k_a + (a - kt_lo) * kTileBytes, q_a, 128);
        umma_commit(&sm.bar_sfull[X]);
      }
      umma_commit(&sm.bar_fin[X]);
      drain_wait(&sm.bar_fin[X], 0);
    }
    __syncwarp();
   }
  } else {
    // ------------------------------------------------------------- softmax
    regs_alloc<kRowsSoftmaxRegs>();
    const int X = warp >> 2;              // warpgroup = query tile of the pair
    const int kloX = X ? klo[1] : klo[0], khiX = X ? khi[1] : khi[0];
    const int wq = warp & 3;              // TMEM lane quarter of this warp
    const int r = tid & 127;              // row inside the tile == TMEM lane
    const int qt = q_first + X;
    const int r0 = qt * kTile;
    const bool active = X == 0 || hasB;
    const int i = r0 + r;                 // current index of this query row
    const uint32_t lane_off = static_cast<uint32_t>(wq * 32) << 16;
    const uint32_t tS = tm + col_s(X) + lane_off, tP = tm + col_p(X) + lane_off,
                   tO = tm + col_o(X) + lane_off;
    bool row_global = false;
    for (int g = 0; g < ng; ++g) row_global |= (sm.gc[g] == i);
    const bool valid = (i < n) && !row_global;
    // allowed band keys of this row, inclusive (current index); the same band
    // is used for rows whose results are discarded (global rows, rows >= n)
    const int lo = max(0, i - p.w);
    const int hi = min(n - 1, i + p.w);

    // lsum: the row sum of the exponentials (fp32), which gives the row's LSE
    // for the column sums; osum: the sum of the same values rounded to the
    // bf16 that P V multiplies, which normalises O (so that O is a weighted
    // mean of V rows whatever the rounding of P)
    float m_ref = -INFINITY, lsum = 0.f, osum = 0.f;
    bool ok = active;
    uint32_t pv_issued = 0;               // P V products issued for this warpgroup

    if (ok && ngp) {
      ok = warp_wait(&sm.bar_sg[X], 0, abort_flag);
      if (ok) {
        float xg[kMaxGlobal];
        tc_fence_after();
        tmem_ld16(tP, xg);                // S_G
        tmem_ld_wait();
        float mx = -INFINITY;
#pragma unroll
        for (int g = 0; g < kMaxGlobal; ++g) {
          const bool use = (g < ng) && abs(i - sm.gc[g]) > p.w;
          xg[g] = use ? xg[g] : -INFINITY;
          mx = fmaxf(mx, xg[g]);
        }
        m_ref = mx * kLogitScale2;
        const float nref = (m_ref == -INFINITY) ? 0.f : -m_ref;
        uint32_t pk[8];
#pragma unroll
        for (int g = 0; g < kMaxGlobal; g += 2) {
          const float a = ex2(fmaf(xg[g], kLogitScale2, nref));
          const float c = ex2(fmaf(xg[g + 1], kLogitScale2, nref));
          pk[g / 2] = pack_bf16x2(a, c);
          lsum += a + c;
          osum = add_bf16_hi(add_bf16_lo(osum, pk[g / 2]), pk[g / 2]);
        }
        tmem_st8(tP + 16, pk);            // P_G
        tmem_st_wait();
        tc_fence_before();
        warp_arrive(&sm.bar_pready[X]);
        pv_issued = 1;
      }
    }

    // Softmax with a running reference m_ref (base-2 units): P = exp2(x - ref).
    // The tile's maximum is taken before its exponentials; when it exceeds the
    // reference by more than 8, the reference is raised and O (all earlier
    // P V complete) and the row sum are rescaled exactly.  P stays below 2^8.
    // All exponentials of the tile are formed in registers before the previous
    // P V is awaited: only the P store and a rescale of O depend on it.
    const uint64_t c2 = f2_pack(kLogitScale2, kLogitScale2);
    for (int t = 0; ok && t <= khiX - kloX; ++t) {
      const int j0 = (kloX + t) * kTile;
      const int a = lo - j0, e = hi - j0;   // this row's allowed columns of the tile
      if (!(ok = warp_wait(&sm.bar_sfull[X], t & 1, abort_flag))) break;
      tc_fence_after();
      float x[128];
#pragma unroll
      for (int ch = 0; ch < 4; ++ch) tmem_ld32(tS + 32 * ch, x + 32 * ch);
      tmem_ld_wait();
      tc_fence_before();
      warp_arrive(&sm.bar_sfree[X]);   // S is in registers: the next S may overwrite it
      // keys outside a row's band take no part; tiles inside the band of all
      // 32 rows of the warp (most of them) need no mask
      if (!__all_sync(0xffffffffu, a <= 0 && e >= kTile - 1)) {
#pragma unroll
        for (int ch = 0; ch < 4; ++ch) {
          // this row's allowed keys among the chunk's 32, as bits; chunks
          // that every row of the warp takes whole are left alone
          const uint32_t keep = bit_range32(a - 32 * ch, e - 32 * ch);
          if (__any_sync(0xffffffffu, keep != 0xffffffffu)) {
#pragma unroll
            for (int k = 0; k < 32; ++k) {
              const uint32_t out =
                  ~static_cast<uint32_t>(static_cast<int32_t>(keep << (31 - k)) >> 31);
              x[32 * ch + k] =
                  __uint_as_float((__float_as_uint(x[32 * ch + k]) & ~out) | (0xff800000u & out));
            }
          }
        }
      }
      float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
      for (int k = 0; k < kTile; k += 8) {
        m4[0] = fmax3(m4[0], x[k], x[k + 1]);
        m4[1] = fmax3(m4[1], x[k + 2], x[k + 3]);
        m4[2] = fmax3(m4[2], x[k + 4], x[k + 5]);
        m4[3] = fmax3(m4[3], x[k + 6], x[k + 7]);
      }
      const float tmax = fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3])) * kLogitScale2;
      const bool raise = tmax > m_ref + 8.f;
      float f = 1.f;
      if (raise) {
        f = (m_ref == -INFINITY) ? 0.f : ex2(m_ref - tmax);
        m_ref = tmax;
        lsum *= f;
        osum *= f;
      }
      const float nref = (m_ref == -INFINITY) ? 0.f : -m_ref;
      const uint64_t n2 = f2_pack(nref, nref);
      uint64_t s2a = f2_pack(0.f, 0.f), s2b = s2a;
      float sq[4] = {0.f, 0.f, 0.f, 0.f};
      uint32_t pk[64];
#pragma unroll
      for (int k = 0; k < kTile; k += 2) {
        float u, w;
        f2_unpack(f2_fma(f2_pack(x[k], x[k + 1]), c2, n2), u, w);
        u = ex2(u);
        w = ex2(w);
        if (k & 2) s2b = f2_add(s2b, f2_pack(u, w));
        else s2a = f2_add(s2a, f2_pack(u, w));
        pk[k >> 1] = pack_bf16x2(u, w);
        const int c = (k >> 1) & 1;
        sq[2 * c] = add_bf16_lo(sq[2 * c], pk[k >> 1]);
        sq[2 * c + 1] = add_bf16_hi(sq[2 * c + 1], pk[k >> 1]);
      }
      float sa, sb, sc2, sd;
      f2_unpack(s2a, sa, sb);
      f2_unpack(s2b, sc2, sd);
      lsum += (sa + sb) + (sc2 + sd);
      osum += (sq[0] + sq[1]) + (sq[2] + sq[3]);
      // every earlier P V has completed: O is final for a rescale and the P
      // columns of this warpgroup are free again
      if (pv_issued > 0 && !(ok = warp_wait(&sm.bar_pvdone[X], (pv_issued - 1) & 1, abort_flag)))
        break;
      tc_fence_after();
      if (__any_sync(0xffffffffu, raise) && pv_issued > 0) {
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
#pragma unroll
      for (int ch = 0; ch < 4; ++ch) tmem_st16(tP + 16 * ch, pk + 16 * ch);
      tmem_st_wait();
      tc_fence_before();
      warp_arrive(&sm.bar_pready[X]);
      ++pv_issued;
    }

    // ---- epilogue: LSE, the global keys and queries, the band's column
    // sums, O
    float lse = INFINITY;
    const bool have_o = ok && pv_issued > 0 &&
                        (ok = warp_wait(&sm.bar_pvdone[X], (pv_issued - 1) & 1, abort_flag));
    if (have_o) lse = valid ? m_ref + lg2(lsum) : INFINITY;
    if (active) sm.nlse[X][r] = -lse;

    if (active && ngp) {
      // Per-warp partial results (32 rows / 32 keys each), reduced with
      // butterfly shuffles and merged later in a fixed order: no barrier here.
      const size_t slot0 =
          (((static_cast<size_t>(b) * p.H + h) * p.T + qt) * 4 + wq) * kMaxGlobal;
      const int gme = lane >> 1;            // global index this lane reports
      const bool writer = (lane & 1) == 0 && gme < ng;
      float xg[kMaxGlobal], xt[kMaxGlobal];
      const bool ok2 = ok && warp_wait(&sm.bar_sgend[X], 0, abort_flag);
      if (ok2) {
        tc_fence_after();
        tmem_ld16(tS, xg);                  // S_G
        tmem_ld16(tS + 16, xt);             // S_Gt
        tmem_ld_wait();
      }
      // S_G and S_Gt are in registers: the S columns take the band pass while
      // the global keys and queries are evaluated
      tc_fence_before();
      warp_arrive(&sm.bar_sfree[X]);
      // far-row column sums of the global keys: rows outside the key's band
      float e16[kMaxGlobal];
#pragma unroll
      for (int g = 0; g < kMaxGlobal; ++g) {
        const bool use = ok2 && valid && g < ng && abs(i - sm.gc[g]) > p.w;
        e16[g] = use ? ex2(fmaf(xg[g], kLogitScale2, -lse)) : 0.f;
      }
      const float gsum = warp_reduce16(e16, OpAdd());
      if (writer) p.gpart[slot0 + gme] = gsum;
      // (max, sum) of each global query over this warp's keys j = 128 qt + r
      const bool key_ok = ok2 && (r0 + r < n);
      float y[kMaxGlobal];
#pragma unroll
      for (int g = 0; g < kMaxGlobal; ++g) {
        y[g] = (key_ok && g < ng) ? xt[g] * kLogitScale2 : -INFINITY;
        e16[g] = y[g];
      }
      const float mme = warp_reduce16(e16, OpMax());
#pragma unroll
      for (int g = 0; g < kMaxGlobal; ++g) {
        const float mg = __shfl_sync(0xffffffffu, mme, 2 * g);
        e16[g] = mg == -INFINITY ? 0.f : ex2(y[g] - mg);
      }
      const float sme = warp_reduce16(e16, OpAdd());
      if (writer) {
        p.gstat[2 * (slot0 + gme)] = mme;
        p.gstat[2 * (slot0 + gme) + 1] = sme;
      }
    }

    // Band pass (the column sums of Sec. "Extractor of Attention Scores"):
    // for each key j of the band, the sum over this tile's rows i of
    // exp2(S_ij scaled - LSE_i); global rows (LSE = +inf) and rows past the
    // end add nothing.  One thread per key column of S^T; written per query
    // tile, summed over query tiles and heads in a fixed order by the
    // finalisation.
    if (active) named_sync_wg(X);   // every -LSE of the tile is in shared memory
    const int nt = khiX - kloX + 1;
    const uint64_t c2b = f2_pack(kLogitScale2, kLogitScale2);
    for (int u = 0; ok && u < nt; ++u) {
      const int j = (kloX + u) * kTile + r;   // key of this thread
      if (!(ok = warp_wait(&sm.bar_sfull[X], (nt + u) & 1, abort_flag))) break;
      tc_fence_after();
      float x[128];
#pragma unroll
      for (int ch = 0; ch < 4; ++ch) tmem_ld32(tS + 32 * ch, x + 32 * ch);
      tmem_ld_wait();
      tc_fence_before();
      warp_arrive(&sm.bar_sfree[X]);   // S^T is in registers
      // query columns r0 + a .. r0 + e are in j's band (and in the sequence)
      const int a = j - p.w - r0, e = min(j + p.w, n - 1) - r0;
      if (!__all_sync(0xffffffffu, a <= 0 && e >= kTile - 1)) {
#pragma unroll
        for (int ch = 0; ch < 4; ++ch) {
          const uint32_t keep = bit_range32(a - 32 * ch, e - 32 * ch);
          if (__any_sync(0xffffffffu, keep != 0xffffffffu)) {
#pragma unroll
            for (int k = 0; k < 32; ++k) {
              const uint32_t out =
                  ~static_cast<uint32_t>(static_cast<int32_t>(keep << (31 - k)) >> 31);
              x[32 * ch + k] =
                  __uint_as_float((__float_as_uint(x[32 * ch + k]) & ~out) | (0xff800000u & out));
            }
          }
        }
      }
      const float* lw = sm.nlse[X];
      uint64_t s2a = f2_pack(0.f, 0.f), s2b = s2a;
#pragma unroll
      for (int k = 0; k < kTile; k += 4) {
        const float4 l4 = *reinterpret_cast<const float4*>(lw + k);
        float e0, e1, e2, e3;
        f2_unpack(f2_fma(f2_pack(x[k], x[k + 1]), c2b, f2_pack(l4.x, l4.y)), e0, e1);
        f2_unpack(f2_fma(f2_pack(x[k + 2], x[k + 3]), c2b, f2_pack(l4.z, l4.w)), e2, e3);
        s2a = f2_add(s2a, f2_pack(ex2(e0), ex2(e1)));
        s2b = f2_add(s2b, f2_pack(ex2(e2), ex2(e3)));
      }
      float sa, sb, sc2, sd;
      f2_unpack(s2a, sa, sb);
      f2_unpack(s2b, sc2, sd);
      if (j < n)
        p.colpart[((static_cast<size_t>(b) * p.H + h) * p.L + j) * band_slots + qt % band_slots] =
            (sa + sc2) + (sb + sd);
    }

    // ---- O: its rows leave through this warp's quarter of its Q tile; every
    // MMA that read the tile completed before the last S^T was awaited
    if (ok && have_o && v.O != nullptr) {
      tc_fence_after();
      const float inv = 1.f / osum;
      uint8_t* stage = Qs + X * kTileBytes + wq * 4096;
#pragma unroll
      for (int c = 0; c < 64; c += 32) {
        float o[32];
        tmem_ld32(tO + c, o);
        tmem_ld_wait();
#pragma unroll
        for (int k = 0; k < 32; k += 8)
          stage_row_piece<8>(stage, (c + k) >> 3,
                          make_uint4(pack_bf16x2(o[k] * inv, o[k + 1] * inv),
                                     pack_bf16x2(o[k + 2] * inv, o[k + 3] * inv),
                                     pack_bf16x2(o[k + 4] * inv, o[k + 5] * inv),
                                     pack_bf16x2(o[k + 6] * inv, o[k + 7] * inv)));
      }
      flush_staged_rows<8>(stage,
                        v.O + ((static_cast<size_t>(b) * p.L + r0 + 32 * wq) * p.H + h) * kHeadDim,
                        static_cast<size_t>(p.H) * kHeadDim, __ballot_sync(0xffffffffu, valid));
    }
  }

  tc_fence_before();
  __threadfence();   // O, the partial sums and statistics of this CTA ...
  __syncthreads();
  if (warp == 9) {
    tc_fence_after();
    tmem_dealloc(tm, 512);
  }
  if (tid == 0) {
    if (sm.abort) atomicOr(p.status, kStatusTimeout);
    red_release_add_u32(p.rows_done + b * p.H + h, 1u);   // ... are visible to the cols CTAs
  }
}

// ---------------------------------------------------------------------------
// cols kernel
// ---------------------------------------------------------------------------
// One CTA per pair of 128-key tiles (2p, 2p+1) of one (sequence, head), one
// warpgroup per key tile.  The band rows' column sums come from the rows
// kernel (one partial per query tile); here: the global rows' P over the
// pair's keys and their P V, the keys' column sums, and the finalisation.
// Tensor memory (256 columns, so that two CTAs share an SM) per warpgroup X:
// S^T against the global queries [16 X, +16), the global rows' P V
// [64 + 64 X, +64).
// The band rows' column sums of key j from the rows kernel, one per query tile
// qlo..qhi in tile order (slot = tile mod kSlots); entries past qhi are 0.
template <int kSlots>
__device__ __forceinline__ void load_band_parts(float (&part)[kWideBandTiles], const LayerParams& p,
                                                int b, int h, int j, int qlo, int qhi, bool use) {
  const float* cp = p.colpart + ((static_cast<size_t>(b) * p.H + h) * p.L + j) * kSlots;
#pragma unroll
  for (int u = 0; u < kWideBandTiles; ++u)
    part[u] = (u < kSlots && use && qlo + u <= qhi) ? __ldcg(cp + (qlo + u) % kSlots) : 0.f;
}

constexpr int kColsThreads = 320;
// The global rows' P is the A operand of an M = 128 MMA whose rows past the 16
// global rows are never used: each 64-key block of that A tile holds its 16
// valid rows (2 KB) and lets the MMA read the following rows from whatever
// shared memory comes next (the K and V tiles), so only 2 KB is reserved.
constexpr uint32_t kPgBlock = 2 * 1024;

struct ColsSmem {
  uint64_t bar_kv;
  uint64_t bar_sfull[2], bar_sfree[2], bar_sg[2], bar_pg[2], bar_og[2], bar_fin;
  uint32_t tmem_base;
  int abort;
  int gc[kMaxGlobal];
  float lse_g[kMaxGlobal];
  int flag, flag2;
  int gnew[kMaxGlobal];
  // each key tile's part of the global rows' P V (warpgroup X), added in
  // tile order into the pair's part
  alignas(16) float ogx[2][kMaxGlobal][kHeadDim];   // read and written as float4
  // sequence compaction: per (round, warp) ballot of kept tokens and the
  // exclusive prefix of their counts
  uint32_t kbits[(kMaxLen + kColsThreads - 1) / kColsThreads][kColsThreads / 32];
  int kpre[(kMaxLen + kColsThreads - 1) / kColsThreads][kColsThreads / 32];
  int last_pos;
  int total;
};

// dynamic shared memory: the global rows' P blocks (2 per warpgroup), K and V
// of both key tiles, the global queries
constexpr uint32_t kColsDyn = 4 * kPgBlock + kTileBytes * 4 + kGTileBytes + 1024;
static_assert(3 * kPgBlock + kTileBytes <= 4 * kPgBlock + 4 * kTileBytes,
              "the A operand's unused rows stay inside the shared memory");

__device__ void finalize_sequence(const LayerParams& p, const LayerView& v, int b, int n,
                                  ColsSmem& sm, uint8_t* scratch);

__global__ void __launch_bounds__(kColsThreads, 2)
    sc_cols_kernel(const __grid_constant__ TensorMaps maps, const __grid_constant__ LayerParams p) {
  // No grid-wide wait on the rows kernel: this kernel is scheduled only after
  // every rows CTA has passed its own wait (so the earlier kernels' results
  // are complete), and each CTA waits below for the rows CTAs of its own
  // (sequence, head) only, so that it can run beside the rows kernel's last CTAs.
  pdl_launch_dependents();
  const int T2 = (p.T + 1) / 2;
  const int pr = blockIdx.x % T2, bh = blockIdx.x / T2;
  const int h = bh % p.H, b = bh / p.H;
  const LayerView v = layer_view(p);
  if (owned_by_tail(p, v, b)) return;
  const int n = __ldcg(v.len + b);
  if (n == 0) {
    if (pr == 0 && h == 0 && threadIdx.x == 0) {
      v.len_out[b] = 0;
      v.ng_out[b] = 0;
      v.ident_out[b] = 1;
    }
    return;
  }
  if (2 * pr * kTile >= n) return;
  const int ng = min(__ldcg(v.ng + b), kMaxGlobal);
  const int ngp = ng > 0 ? kMaxGlobal : 0;
  const int Tn = (n + kTile - 1) / kTile;
  const int Tp = (Tn + 1) / 2;
  const bool hasB = (2 * pr + 1) * kTile < n;

  extern __shared__ uint8_t dyn_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dyn_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* Pg = base;                              // 2 x 2 blocks of 16 rows
  uint8_t* Ks = Pg + 4 * kPgBlock;                 // 2 tiles
  uint8_t* Vs = Ks + 2 * kTileBytes;               // 2 tiles
  uint8_t* QG = Vs + 2 * kTileBytes;
  __shared__ ColsSmem sm;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  int qlo[2], qhi[2];
#pragma unroll
  for (int X = 0; X < 2; ++X) {
    const int j0 = (2 * pr + X) * kTile, j1 = min(j0 + kTile - 1, n - 1);
    qlo[X] = max(0, j0 - p.w) / kTile;
    qhi[X] = min(n - 1, j1 + p.w) / kTile;
  }

  if (tid == 0) {
    mbar_init(&sm.bar_kv, 1);
    for (int X = 0; X < 2; ++X) {
      mbar_init(&sm.bar_sfull[X], 1);
      mbar_init(&sm.bar_sfree[X], 4);   // one arrival per warp
      mbar_init(&sm.bar_sg[X], 1);
      mbar_init(&sm.bar_pg[X], 4);
      mbar_init(&sm.bar_og[X], 1);
    }
    mbar_init(&sm.bar_fin, 1);
    sm.abort = 0;
    fence_mbar_init();
  }
  if (tid < kMaxGlobal) sm.gc[tid] = tid < ng ? __ldcg(v.gcur + b * kMaxGlobal + tid) : -1;
  if (warp == 9) tmem_alloc(&sm.tmem_base, 256);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = sm.tmem_base;
  volatile int* abort_flag = &sm.abort;

  if (warp == 8) {
    const RowSource rs = row_source(p, v, b);
    // this sequence's rows may still be crossing the host link
    if (p.gathered != nullptr) {
      if (lane == 0) wait_count(p.gathered + b, p.gather_target, abort_flag);
      __syncwarp();
      fence_proxy_async_global();
    }
    if (lane == 0) {
      mbar_arrive_expect_tx(&sm.bar_kv, (hasB ? 4 : 2) * kTileBytes + ngp * 128);
      for (int X = 0; X < (hasB ? 2 : 1); ++X) {
        load_tile(maps, 1, rs, h, (2 * pr + X) * kTile, Ks + X * kTileBytes, &sm.bar_kv);
        load_tile(maps, 2, rs, h, (2 * pr + X) * kTile, Vs + X * kTileBytes, &sm.bar_kv);
      }
    }
    __syncwarp();
    if (ngp) load_globals(maps, 0, rs, h, p.H, sm.gc, ng, QG, &sm.bar_kv, lane);
    if (lane == 0) drain_wait(&sm.bar_kv, 0);
  } else if (warp == 9) {
    if (lane == 0) {
      const uint32_t k_a = smem_u32(Ks), v_a = smem_u32(Vs);
      const int nX = hasB ? 2 : 1;
      bool ok = mbar_wait(&sm.bar_kv, 0, abort_flag);
      if (ok) {
        tc_fence_after();
        if (ngp)
          for (int X = 0; X < nX; ++X) {
            mma_qk(tm + 16 * X, k_a + X * kTileBytes, smem_u32(QG), 16);
            umma_commit(&sm.bar_sg[X]);
          }
      }
      if (ok && ngp)
        for (int X = 0; ok && X < nX; ++X) {
          if (!(ok = mbar_wait(&sm.bar_pg[X], 0, abort_flag))) break;
          tc_fence_after();
          mma_pv(tm + 64 + 64 * X, smem_u32(Pg) + X * 2 * kPgBlock, kPgBlock, v_a + X * kTileBytes,
                 kTile / 16, false);
          umma_commit(&sm.bar_og[X]);
        }
      umma_commit(&sm.bar_fin);
      drain_wait(&sm.bar_fin, 0);
    }
    __syncwarp();
  } else {
    const int X = warp >> 2, wq = warp & 3;
    const int qloX = X ? qlo[1] : qlo[0], qhiX = X ? qhi[1] : qhi[0];
    const int r = tid & 127;
    const int kt = 2 * pr + X;
    const int j0 = kt * kTile;
    const int j = j0 + r;             // key column owned by this thread
    const bool active = X == 0 || hasB;
    const uint32_t lane_off = static_cast<uint32_t>(wq * 32) << 16;
    const uint32_t tSG = tm + 16 * X, tOG = tm + 64 + 64 * X;
    // the rows CTAs of this (sequence, head) have finished (their partial
    // sums, statistics and the cleared global-row outputs are read below)
    if (tid == 0)
      wait_count(p.rows_done + b * p.H + h,
                 static_cast<uint32_t>((p.wide || p.band) ? Tn : Tp), abort_flag);
    asm volatile("bar.sync 3, 256;" ::: "memory");
    // every load of the prologue is issued before any is used: this key's
    // band-row column sums of the query tiles of its band (one per tile, from
    // the rows kernel) and, per warp, the (max, sum) pieces of global rows
    // warp and warp + 8
    float part[kWideBandTiles];
    if (p.band_slots == kMaxBandTiles)
      load_band_parts<kMaxBandTiles>(part, p, b, h, j, qloX, qhiX, active && j < n);
    else
      load_band_parts<kWideBandTiles>(part, p, b, h, j, qloX, qhiX, active && j < n);
    // lane k takes entries k, k+32, k+64, k+96 of the 4 Tn (key tile, warp
    // slice) pieces; the warp combines them in a fixed order
    const size_t base_slot = (static_cast<size_t>(b) * p.H + h) * p.T * 4 * kMaxGlobal;
    float me[2][4], se[2][4];
    // the far-row sums (rows whose band does not reach the key) of a global
    // key among this warp's 32 keys, over the (query tile, warp slice) pieces
    // of this head: lane k loads pieces k, k+32, k+64, k+96 (at most one
    // global key per warp is usual; more are summed one after another below)
    const int wk0 = j0 + 32 * wq;
    float far[4] = {0.f, 0.f, 0.f, 0.f};
    int far_g = -1;
    if (active && ngp) {
#pragma unroll 1
      for (int g = 0; g < ng; ++g)
        if (sm.gc[g] >= wk0 && sm.gc[g] < wk0 + 32) {
          far_g = g;
          break;
        }
      if (far_g >= 0) {
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const int ent = lane + 32 * k;
          far[k] = ent < 4 * Tn ? __ldcg(p.gpart + base_slot + ent * kMaxGlobal + far_g) : 0.f;
        }
      }
    }
#pragma unroll
    for (int gg = 0; gg < 2; ++gg) {
      const int g = warp + 8 * gg;
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int ent = lane + 32 * k;
        const bool use = ngp && g < ng && ent < 4 * Tn;
        me[gg][k] = use ? __ldcg(p.gstat + 2 * (base_slot + ent * kMaxGlobal + g)) : -INFINITY;
        se[gg][k] = use ? __ldcg(p.gstat + 2 * (base_slot + ent * kMaxGlobal + g) + 1) : 0.f;
      }
    }
#pragma unroll
    for (int gg = 0; gg < 2; ++gg) {
      const int g = warp + 8 * gg;
      if (!ngp || g >= ng) continue;   // warp-uniform
      const float m = fmaxf(fmaxf(me[gg][0], me[gg][1]), fmaxf(me[gg][2], me[gg][3]));
      float sacc = 0.f;
#pragma unroll
      for (int k = 0; k < 4; ++k)
        sacc += (me[gg][k] == -INFINITY) ? 0.f : se[gg][k] * ex2(me[gg][k] - m);
      const float M = warp_max(m);
      const float S = warp_sum(m == -INFINITY ? 0.f : sacc * ex2(m - M));
      if (lane == 0) sm.lse_g[g] = M + lg2(S);
    }
    asm volatile("bar.sync 3, 256;" ::: "memory");

    // band rows: the query tiles' sums in tile order
    float acc = 0.f;
#pragma unroll
    for (int u = 0; u < kWideBandTiles; ++u) acc += part[u];
    // far rows of the global keys among this warp's keys (gc increases with
    // g, so they are consecutive entries of the list)
    if (far_g >= 0) {
#pragma unroll 1
      for (int g = far_g; g < ng; ++g) {
        const int cg = sm.gc[g];
        if (cg >= wk0 + 32) break;
        if (g != far_g) {
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const int ent = lane + 32 * k;
            far[k] = ent < 4 * Tn ? __ldcg(p.gpart + base_slot + ent * kMaxGlobal + g) : 0.f;
          }
        }
        const float fs = warp_sum((far[0] + far[1]) + (far[2] + far[3]));
        if (j == cg) acc += fs;
      }
    }
    const bool ok = active;
    float x[16];

    if (active && ngp) {
      bool ok2 = ok && warp_wait(&sm.bar_sg[X], 0, abort_flag);
      if (ok2) {
        tc_fence_after();
        tmem_ld16(tSG + lane_off, x);
        tmem_ld_wait();
      }
      uint16_t pb[kMaxGlobal];
      float s = 0.f;
#pragma unroll
      for (int g = 0; g < kMaxGlobal; ++g) {
        const float v =
            (ok2 && g < ng && j < n) ? ex2(fmaf(x[g], kLogitScale2, -sm.lse_g[g])) : 0.f;
        s += v;
        pb[g] = __bfloat16_as_ushort(__float2bfloat16_rn(v));
      }
      acc += s;
      // P of the global rows, transposed into this warpgroup's A tile: row g,
      // column (key) r
      uint8_t* col = Pg + X * 2 * kPgBlock + (r >> 6) * kPgBlock;
      const int ch = (r & 63) >> 3, wi = (r & 7) * 2;
#pragma unroll
      for (int g = 0; g < kMaxGlobal; ++g)
        *reinterpret_cast<uint16_t*>(col + sw128_offset(g, ch) + wi) = pb[g];
      fence_proxy_async_smem();
      tc_fence_before();
      warp_arrive(&sm.bar_pg[X]);
      bool ok3 = ok2 && warp_wait(&sm.bar_og[X], 0, abort_flag);
      if (wq == 0) {
        // this key tile's part of the global rows' outputs (TMEM lane g = global g)
        if (ok3) tc_fence_after();
        float* mine = &sm.ogx[X][lane & (kMaxGlobal - 1)][0];
#pragma unroll 1
        for (int c = 0; c < 64; c += 16) {
          float o[16];
          if (ok3) {
            tmem_ld16(tOG + lane_off + c, o);
            tmem_ld_wait();
          } else {
#pragma unroll
            for (int k = 0; k < 16; ++k) o[k] = 0.f;
          }
          if (lane < kMaxGlobal)
#pragma unroll
            for (int k = 0; k < 16; k += 4)
              *reinterpret_cast<float4*>(mine + c + k) = make_float4(o[k], o[k + 1], o[k + 2], o[k + 3]);
        }
        // warps 0 and 4 (the first warp of each warpgroup) meet here when the
        // pair has two key tiles; warp 0 adds the parts in tile order and
        // stores the pair's part (plain stores: no order-dependent atomics)
        if (hasB) asm volatile("bar.sync 5, 64;" ::: "memory");
        else __syncwarp();
        if (X == 0) {
          float* part = p.og + (((static_cast<size_t>(b) * p.H + h) * T2 + pr) * kMaxGlobal) *
                                   kHeadDim;
          for (int k = lane; k < ng * (kHeadDim / 4); k += 32) {
            const int g = k / (kHeadDim / 4), d = 4 * (k % (kHeadDim / 4));
            float4 a4 = *reinterpret_cast<const float4*>(&sm.ogx[0][g][d]);
            if (hasB) {
              const float4 b4 = *reinterpret_cast<const float4*>(&sm.ogx[1][g][d]);
              a4.x += b4.x; a4.y += b4.y; a4.z += b4.z; a4.w += b4.w;
            }
            *reinterpret_cast<float4*>(part + g * kHeadDim + d) = a4;
          }
        }
      }
    }
    if (active && j < n) p.acc[(static_cast<size_t>(b) * p.H + h) * p.L + j] = acc;
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 9) {
    tc_fence_after();
    tmem_dealloc(tm, 256);
  }
  if (tid == 0 && sm.abort) atomicOr(p.status, kStatusTimeout);

  // One hand-over for both roles below: this CTA's part of the global rows'
  // outputs and its column sums are visible before either counter is raised.
  __threadfence();
  __syncthreads();
  if (tid == 0) {
    sm.flag = ngp && atomicAdd(p.cols_done + b * p.H + h, 1u) == static_cast<uint32_t>(Tp - 1);
    sm.flag2 = atomicAdd(p.cnt_tile + b * p.T + pr, 1u) == static_cast<uint32_t>(p.H - 1);
  }
  __syncthreads();

  // ---- last pair of this (sequence, head): the global rows' outputs, the
  // pairs' parts added in pair order
  if (ngp) {
    if (sm.flag) {
      __threadfence();
      const float* part0 =
          p.og + (static_cast<size_t>(b) * p.H + h) * T2 * kMaxGlobal * kHeadDim;
      for (int k = tid; k < ng * (kHeadDim / 4); k += kColsThreads) {
        const int g = k / (kHeadDim / 4), d = 4 * (k % (kHeadDim / 4));
        constexpr int kBatch = 8;   // loads in flight before they are added
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int q0 = 0; q0 < Tp; q0 += kBatch) {
          float4 x[kBatch];
#pragma unroll
          for (int u = 0; u < kBatch; ++u)
            x[u] = q0 + u < Tp ? __ldcg(reinterpret_cast<const float4*>(
                                     part0 + ((q0 + u) * kMaxGlobal + g) * kHeadDim + d))
                               : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
          for (int u = 0; u < kBatch; ++u) {
            acc.x += x[u].x; acc.y += x[u].y; acc.z += x[u].z; acc.w += x[u].w;
          }
        }
        if (v.O != nullptr)
          *reinterpret_cast<uint2*>(v.O + ((static_cast<size_t>(b) * p.L + sm.gc[g]) * p.H + h) *
                                              kHeadDim + d) =
              make_uint2(pack_bf16x2(acc.x, acc.y), pack_bf16x2(acc.z, acc.w));
      }
      if (tid == 0) p.cols_done[b * p.H + h] = 0u;
    }
  }

  // ---- last head of this pair of key tiles: scores and keep flags (fixed head order)
  if (!sm.flag2) return;
  __threadfence();
  const int j0 = 2 * pr * kTile;
  const int jn = min(n, j0 + 2 * kTile);
  // this thread's key column: every head's column sum, loaded first (in
  // flight while the global keys' partial sums are reduced below)
  const int jj = j0 + tid;
  const bool my_key = tid < 2 * kTile && jj < jn;
  float hs[kTailMaxHeads];
  float a = 0.f;
  const float* ap = p.acc + static_cast<size_t>(b) * p.H * p.L + jj;
#pragma unroll
  for (int u = 0; u < kTailMaxHeads; ++u)
    hs[u] = my_key && u < p.H ? __ldcg(ap + static_cast<size_t>(u) * p.L) : 0.f;
  for (int h0 = kTailMaxHeads; my_key && h0 < p.H; ++h0)   // more than 16 heads
    a += __ldcg(ap + static_cast<size_t>(h0) * p.L);
  if (my_key) {
    float hsum = 0.f;
#pragma unroll
    for (int u = 0; u < kTailMaxHeads; ++u) hsum += hs[u];   // heads in order
    a = hsum + a;
    const float s = a / static_cast<float>(p.H * n);
    v.scores[static_cast<size_t>(b) * p.L + jj] = s;
    if (p.keep_rule != kKeepTopRatio) {   // the top-ratio cut needs every score first
      const float theta = p.theta ? __ldg(p.theta + b)
                          : p.keep_rule == kKeepAbsolute ? v.alpha
                                                         : v.alpha / static_cast<float>(n);
      p.keep[static_cast<size_t>(b) * p.L + jj] = (jj == 0 || s >= theta) ? 1 : 0;
    }
  }
  if (tid == 0) p.cnt_tile[b * p.T + pr] = 0u;
  __threadfence();
  __syncthreads();
  if (tid == 0) sm.flag = (atomicAdd(p.cnt_seq + b, 1u) == static_cast<uint32_t>(Tp - 1));
  __syncthreads();
  if (!sm.flag) return;
  __threadfence();
  finalize_sequence(p, v, b, n, sm, base);
}

struct BlockSync {
  __device__ __forceinline__ void operator()() const { __syncthreads(); }
};

// Order-preserving compaction of sequence b's kept tokens, the next layer's
// global list, and the bf16 outputs of the global rows.  One CTA; token c is
// handled by thread c % kColsThreads in round c / kColsThreads (coalesced
// loads, all issued at once); output slots come from warp ballots and a
// fixed-order prefix over (round, warp).  Under the top-ratio rule the keep
// flags come from the cut over all n scores, found here (`scratch`: shared
// memory the CTA no longer uses, for the selection's histogram and tie flags).
__device__ void finalize_sequence(const LayerParams& p, const LayerView& v, int b, int n,
                                  ColsSmem& sm, uint8_t* scratch) {
  constexpr int kRounds = (kMaxLen + kColsThreads - 1) / kColsThreads;
  constexpr int kWarps = kColsThreads / 32;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint8_t* keep = p.keep + static_cast<size_t>(b) * p.L;
  const int32_t* pos = v.pos + static_cast<size_t>(b) * p.L;
  int32_t* pos_out = v.pos_out + static_cast<size_t>(b) * p.L;
  bool kf[kRounds];
  int32_t ps[kRounds];
  if (p.keep_rule == kKeepTopRatio) {
    const float* sc = v.scores + static_cast<size_t>(b) * p.L;
    uint32_t key[kRounds];
#pragma unroll
    for (int r = 0; r < kRounds; ++r) {
      const int c = r * kColsThreads + tid;
      key[r] = (c >= 1 && c < n) ? select_key(__ldcg(sc + c)) : 0u;
      ps[r] = c < n ? __ldcg(pos + c) : 0;
    }
    SelectSmem& ss = *reinterpret_cast<SelectSmem*>(scratch);
    uint8_t* tie = scratch + sizeof(SelectSmem);
    uint32_t cut;
    int ties, eq;
    radix_cut<kColsThreads, kRounds>(key, top_count(v.alpha, n) - 1, n - 1, ss, tid, BlockSync(),
                                     cut, ties, eq);
    const bool split = eq > ties;   // an exact tie straddles the cut
    if (split) rank_ties<kColsThreads, kRounds>(key, cut, ties, n, tie, tid, BlockSync());
#pragma unroll
    for (int r = 0; r < kRounds; ++r) {
      const int c = r * kColsThreads + tid;
      kf[r] = c < n && (c == 0 || key[r] > cut || (key[r] == cut && (!split || tie[c] == 2)));
    }
  } else {
#pragma unroll
    for (int r = 0; r < kRounds; ++r) {
      const int c = r * kColsThreads + tid;
      kf[r] = c < n && __ldcg(keep + c) != 0;
      ps[r] = c < n ? __ldcg(pos + c) : 0;
    }
  }
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    const uint32_t bits = __ballot_sync(0xffffffffu, kf[r]);
    if (lane == 0) sm.kbits[r][warp] = bits;
  }
  if (tid < kMaxGlobal) sm.gnew[tid] = -1;
  __syncthreads();
  if (warp == 0) {
    // prefix over (round, warp) in order: lane l covers entries l, l+32, ...
    constexpr int kEntries = kRounds * kWarps;
    int cnt[(kEntries + 31) / 32];
    int run = 0;
#pragma unroll
    for (int u = 0; u < (kEntries + 31) / 32; ++u) {
      const int e = u * 32 + lane;
      cnt[u] = e < kEntries ? __popc(sm.kbits[e / kWarps][e % kWarps]) : 0;
    }
#pragma unroll
    for (int u = 0; u < (kEntries + 31) / 32; ++u) {
      int x = cnt[u];
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, off);
        if (lane >= off) x += y;
      }
      const int e = u * 32 + lane;
      if (e < kEntries) sm.kpre[e / kWarps][e % kWarps] = run + x - cnt[u];
      run += __shfl_sync(0xffffffffu, x, 31);
    }
    if (lane == 0) sm.total = run;
  }
  __syncthreads();
  const uint32_t below = (1u << lane) - 1u;
#pragma unroll
  for (int r = 0; r < kRounds; ++r) {
    if (!kf[r]) continue;
    const int out = sm.kpre[r][warp] + __popc(sm.kbits[r][warp] & below);
    pos_out[out] = ps[r];
    if (p.kept_cur) p.kept_cur[static_cast<size_t>(b) * p.L + out] = r * kColsThreads + tid;
    if (out == sm.total - 1) sm.last_pos = ps[r];
  }
  // next-layer index of each surviving global token
  const int ng = min(__ldcg(v.ng + b), kMaxGlobal);
  if (tid < ng) {
    const int c = sm.gc[tid], r = c / kColsThreads, t = c % kColsThreads;
    const uint32_t bits = sm.kbits[r][t >> 5];
    if ((bits >> (t & 31)) & 1u) sm.gnew[tid] = sm.kpre[r][t >> 5] + __popc(bits & ((1u << (t & 31)) - 1u));
  }
  __syncthreads();
  if (tid == 0) {
    const int total = sm.total;
    int m = 0;
    for (int g = 0; g < ng; ++g)
      if (sm.gnew[g] >= 0) v.gcur_out[b * kMaxGlobal + m++] = sm.gnew[g];
    v.ng_out[b] = m;
    v.len_out[b] = total;
    if (p.tail_from != nullptr && total <= p.tail_max) p.tail_from[b] = v.layer + 1;
    // the survivors are original positions 0..total-1 exactly when the last one is total-1
    v.ident_out[b] = (!p.no_ident && (total == 0 || sm.last_pos == total - 1)) ? 1 : 0;
    p.cnt_seq[b] = 0u;
    for (int hh = 0; hh < p.H; ++hh) p.rows_done[b * p.H + hh] = 0u;
  }
}

// ---------------------------------------------------------------------------
// gather kernel: the next layer's Q, K, V rows of the kept tokens, compacted
// ---------------------------------------------------------------------------
constexpr int kGatherTokens = 8;
constexpr int kGatherThreads = 256;

// One item: tokens 8 ch .. 8 ch + 7 of sequence b, 3 tensors; with H = 12 each
// thread moves at most nine 16-byte vectors, all loads issued before any store.
__device__ __forceinline__ void gather_item(const GatherParams& g, int b, int ch, int layer,
                                            long long src_base, const int32_t* lenp,
                                            const int32_t* posp, const int32_t* identp) {
  if (g.tail_from != nullptr && __ldcg(g.tail_from + b) <= layer) return;
  const int n = __ldcg(lenp + b);
  const int c0 = ch * kGatherTokens;
  if (__ldcg(identp + b) != 0 || c0 >= n) return;
  const int cnt = min(kGatherTokens, n - c0);
  const int vec = g.H * kHeadDim / 8;  // 16-byte vectors per token row
  const int total = cnt * vec;
  const long long dst_tok0 = static_cast<long long>(b) * g.L + c0;
  const long long src_tok0 = src_base + static_cast<long long>(b) * g.L;
  constexpr int kPer = 4;   // vectors per thread and tensor per round
  for (int k0 = threadIdx.x; k0 < total; k0 += kGatherThreads * kPer) {
    uint4 v[3][kPer];
    long long so[kPer], doff[kPer];
#pragma unroll
    for (int u = 0; u < kPer; ++u) {
      const int k = k0 + u * kGatherThreads;
      const int tk = k / vec, e = k - tk * vec;
      so[u] = k < total ? (src_tok0 + __ldcg(posp + static_cast<size_t>(b) * g.L + c0 + tk)) * vec + e
                        : -1;
      doff[u] = (dst_tok0 + tk) * vec + e;
    }
#pragma unroll
    for (int t = 0; t < 3; ++t)
#pragma unroll
      for (int u = 0; u < kPer; ++u)
        if (so[u] >= 0) v[t][u] = __ldg(reinterpret_cast<const uint4*>(g.src[t]) + so[u]);
#pragma unroll
    for (int t = 0; t < 3; ++t)
#pragma unroll
      for (int u = 0; u < kPer; ++u)
        if (so[u] >= 0) reinterpret_cast<uint4*>(g.dst[t])[doff[u]] = v[t][u];
  }
}

// The per-layer gather: one CTA per item (grid: chunks x sequences).
__global__ void __launch_bounds__(kGatherThreads)
    sc_gather_kernel(const GatherParams g) {
  pdl_launch_dependents();
  pdl_wait();
  int layer = g.layer;
  long long src_base = g.src_base;
  const int32_t* lenp = g.len;
  const int32_t* posp = g.pos;
  const int32_t* identp = g.ident;
  if (g.dev_layer != nullptr) {
    layer = __ldcg(g.dev_layer) + 1;
    if (layer >= g.n_layers) return;
    src_base = layer * g.tok_stride;
    lenp += static_cast<size_t>(layer) * g.len_stride;
    posp += layer * g.row_stride;
    identp = g.ident_slot[layer & 1];
  }
  gather_item(g, blockIdx.y, blockIdx.x, layer, src_base, lenp, posp, identp);
}

// The gather with per-sequence counts (g.gathered): a grid-stride walk over
// the items sequence by sequence; gathered[b] is raised (release) once an item
// of sequence b is copied.  Its successor is launched once every CTA has
// passed the grid wait, so what the kernels before this one wrote is complete
// by then.  Used for the layer (given explicitly) whose rows cross the host link.
__global__ void __launch_bounds__(kGatherThreads)
    sc_gather_seq_kernel(const GatherParams g) {
  pdl_wait();
  pdl_launch_dependents();
  const int nch = (g.L + kGatherTokens - 1) / kGatherTokens;
  for (int it = blockIdx.x; it < g.B * nch; it += gridDim.x) {
    const int b = it / nch;
    gather_item(g, b, it - b * nch, g.layer, g.src_base, g.len, g.pos, g.ident);
    __syncthreads();   // every copy of the item is stored ...
    if (threadIdx.x == 0) {
      __threadfence();
      red_release_add_u32(g.gathered + b, 1u);   // ... before it is counted
    }
  }
}

// ---------------------------------------------------------------------------
// export kernel: a stack's results to page-locked host memory
// ---------------------------------------------------------------------------
constexpr int kExportTokens = 32;
constexpr int kExportThreads = 256;

// Work items of 32 current slots of one (layer, sequence), walked by a
// grid-stride loop; only the slots below the layer's length are copied.  Loads
// from device memory are issued in groups of four before the stores, which
// cross the host link.
__global__ void __launch_bounds__(kExportThreads)
    sc_export_kernel(const ExportParams e) {
  // part 1 runs beside the cluster kernel, which lets it start once every one
  // of its CTAs has passed its own grid wait: what part 1 reads is complete
  if (e.part != 1) pdl_wait();
  const int nch = (e.L + kExportTokens - 1) / kExportTokens;
  const int items = (e.n_layers + 1) * e.B * nch;
  const int vec = e.H * kHeadDim / 8;   // 16-byte vectors per row
  for (int it = blockIdx.x; it < items; it += gridDim.x) {
    const int ch = it % nch, lb = it / nch;
    const int b = lb % e.B, l = lb / e.B;
    if (e.part != 0 && (e.part == 1) != (l < __ldcg(e.tail_from + b))) continue;
    const size_t li = static_cast<size_t>(l) * e.B + b;
    const int n = __ldcg(e.len + li);
    if (ch == 0 && threadIdx.x == 0) e.hlen[li] = n;
    const int c0 = ch * kExportTokens;
    if (c0 >= n) continue;
    const int cnt = min(kExportTokens, n - c0);
    const size_t row0 = li * e.L + c0;
    if (threadIdx.x < cnt) {
      e.hpos[row0 + threadIdx.x] = __ldcg(e.pos + row0 + threadIdx.x);
      if (l < e.n_layers) e.hscores[row0 + threadIdx.x] = __ldcg(e.scores + row0 + threadIdx.x);
    }
    if (l >= e.n_layers) continue;
    uint4* dst;
    if (e.hO != nullptr) dst = reinterpret_cast<uint4*>(e.hO) + row0 * vec;
    else if (l == e.n_layers - 1 && e.hO_last != nullptr)
      dst = reinterpret_cast<uint4*>(e.hO_last) + (static_cast<size_t>(b) * e.L + c0) * vec;
    else continue;
    const int total = cnt * vec;
    const uint4* src = reinterpret_cast<const uint4*>(e.O) + row0 * vec;
    constexpr int kPer = 4;
    for (int k0 = threadIdx.x; k0 < total; k0 += kExportThreads * kPer) {
      uint4 v[kPer];
#pragma unroll
      for (int u = 0; u < kPer; ++u) {
        const int k = k0 + u * kExportThreads;
        if (k < total) v[u] = __ldcg(src + k);
      }
#pragma unroll
      for (int u = 0; u < kPer; ++u) {
        const int k = k0 + u * kExportThreads;
        if (k < total) dst[k] = v[u];
      }
    }
  }
  // part 1 completes only after the cluster kernel (which writes its own
  // layers' results to the host buffers), so that the call's last kernel
  // ends after every result is written
  if (e.part == 1) pdl_wait();
}

// ---------------------------------------------------------------------------
// prep kernel: padding removal (stack) or global-token lookup (single layer)
// ---------------------------------------------------------------------------
constexpr int kPrepThreads = 1024;

__global__ void __launch_bounds__(kPrepThreads)
    sc_prep_kernel(const PrepParams pp) {
  pdl_launch_dependents();
  pdl_wait();
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  __shared__ int wsum[kPrepThreads / 32];
  __shared__ int spos[kMaxLen];
  __shared__ int gfound[kMaxGlobal];
  __shared__ int s_n;
  if (pp.pos_in == nullptr) {
    const int L = pp.L;
    int32_t* out = pp.pos_out + static_cast<size_t>(b) * L;
    if (pp.pad_mask == nullptr) {
      // no padding: the current tokens are positions 0..L-1
      for (int c = tid; c < L; c += kPrepThreads) {
        out[c] = c;
        spos[c] = c;
      }
      if (tid == 0) {
        s_n = L;
        pp.len_out[b] = L;
      }
    } else {
      // stack mode with padding: the real tokens in order; thread tid takes
      // one contiguous run, runs are placed by a scan of their counts
      const uint8_t* mask = pp.pad_mask + static_cast<size_t>(b) * L;
      const int per = (L + kPrepThreads - 1) / kPrepThreads;
      const int c0 = min(L, tid * per), c1 = min(L, c0 + per);
      int cnt = 0;
      for (int c = c0; c < c1; ++c) cnt += mask[c] != 0;
      int x = cnt;   // inclusive scan within the warp
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, off);
        if (lane >= off) x += y;
      }
      if (lane == 31) wsum[warp] = x;
      __syncthreads();
      if (warp == 0) {
        int w = wsum[lane];
#pragma unroll
        for (int off = 1; off < 32; off <<= 1) {
          const int y = __shfl_up_sync(0xffffffffu, w, off);
          if (lane >= off) w += y;
        }
        wsum[lane] = w;
      }
      __syncthreads();
      int at = (warp > 0 ? wsum[warp - 1] : 0) + x - cnt;
      for (int c = c0; c < c1; ++c) {
        if (!mask[c]) continue;
        out[at] = c;
        spos[at] = c;
        ++at;
      }
      if (tid == 0) {
        s_n = wsum[kPrepThreads / 32 - 1];
        pp.len_out[b] = s_n;
      }
    }
  } else {
    if (tid == 0) s_n = pp.len_in[b];
    __syncthreads();
    for (int c = tid; c < s_n; c += kPrepThreads)
      spos[c] = pp.pos_in[static_cast<size_t>(b) * pp.L + c];
  }
  __syncthreads();
  const int n = s_n;
  // current index of each global position (one thread each; binary search:
  // positions increase with the current index)
  if (tid < kMaxGlobal) {
    int found = -1;
    if (tid < pp.n_global) {
      const int target = pp.global_pos[tid];
      int lo = 0, hi = n - 1;
      while (lo <= hi) {
        const int mid = (lo + hi) >> 1;
        if (spos[mid] < target) lo = mid + 1;
        else hi = mid - 1;
      }
      if (lo < n && spos[lo] == target) found = lo;
    }
    gfound[tid] = found;
  }
  __syncthreads();
  if (tid == 0) {
    // global positions are sorted, so the matches come out in increasing order
    int m = 0;
    for (int g = 0; g < kMaxGlobal; ++g)
      if (gfound[g] >= 0) pp.gcur[b * kMaxGlobal + m++] = gfound[g];
    pp.ng[b] = m;
    // single-layer calls read their (already current-order) inputs in place
    pp.ident[b] = (!pp.no_ident && (pp.pos_in != nullptr || n == 0 || spos[n - 1] == n - 1))
                      ? 1 : 0;
    if (pp.tail_from != nullptr) pp.tail_from[b] = n <= pp.tail_max ? 0 : 0x7fffffff;
    if (pp.has_cond && n > pp.tail_max) cudaGraphSetConditional(pp.cond, 1u);
    if (pp.dev_layer != nullptr && b == 0) *pp.dev_layer = 0;
  }
}

// ---------------------------------------------------------------------------
// advance kernel: one step of the device-driven layer loop
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) sc_advance_kernel(const AdvanceParams a) {
  pdl_launch_dependents();
  pdl_wait();
  __shared__ int s_layer;
  if (threadIdx.x == 0) s_layer = __ldcg(a.dev_layer) + 1;
  __syncthreads();
  const int l = s_layer;
  int big = 0;
  for (int b = threadIdx.x; b < a.B; b += blockDim.x) big |= __ldcg(a.tail_from + b) > l;
  big = __syncthreads_or(big);
  if (threadIdx.x == 0) {
    *a.dev_layer = l;
    cudaGraphSetConditional(a.cond, (big && l < a.n_layers) ? 1u : 0u);
  }
}

}  // namespace sc

// ---------------------------------------------------------------------------
// launch helpers used by the C ABI
// ---------------------------------------------------------------------------
namespace sc {

// Every kernel of the chain is launched with programmatic stream serialisation:
// it may be scheduled while its predecessor finishes and waits for it on the
// device (pdl_wait) before touching global memory.
template <typename... KArgs, typename... Args>
static cudaError_t launch_chained(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                                  cudaStream_t st, Args&&... args) {
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
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

cudaError_t launch_prep(const PrepParams& pp, cudaStream_t st) {
  return launch_chained(sc_prep_kernel, dim3(pp.B), dim3(kPrepThreads), 0, st, pp);
}

cudaError_t configure_band();

cudaError_t configure_kernels() {
  // the attention kernels use most of an SM's shared memory
  cudaError_t e = configure_band();
  for (auto k : {sc_rows_kernel<false>, sc_rows_kernel<true>}) {
    // the warpgroups' register split (setmaxnreg) needs the whole launch
    // allocation: with fewer registers a thread, an increase would never be granted
    cudaFuncAttributes fa;
    if (e == cudaSuccess) e = cudaFuncGetAttributes(&fa, k);
    if (e == cudaSuccess && fa.numRegs < kRowsLaunchRegs) e = cudaErrorInvalidConfiguration;
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(kRowsDyn));
    if (e == cudaSuccess)
      e = cudaFuncSetAttribute(k, cudaFuncAttributePreferredSharedMemoryCarveout,
                               cudaSharedmemCarveoutMaxShared);
  }
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(sc_cols_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(kColsDyn));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(sc_cols_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                             cudaSharedmemCarveoutMaxShared);
  return e;
}

cudaError_t launch_band(const TensorMaps& m, const LayerParams& p, int sms, cudaStream_t st);

cudaError_t launch_rows(const TensorMaps& m, const LayerParams& p, cudaStream_t st) {
  if (p.band) return launch_band(m, p, p.sms, st);
  if (p.wide)
    return launch_chained(sc_rows_kernel<true>, dim3(p.B * p.H * p.T), dim3(kRowsThreads),
                          kRowsDyn, st, m, p);
  return launch_chained(sc_rows_kernel<false>, dim3(p.B * p.H * ((p.T + 1) / 2)),
                        dim3(kRowsThreads), kRowsDyn, st, m, p);
}

cudaError_t launch_cols(const TensorMaps& m, const LayerParams& p, cudaStream_t st) {
  dim3 grid(p.B * p.H * ((p.T + 1) / 2));
  return launch_chained(sc_cols_kernel, grid, dim3(kColsThreads), kColsDyn, st, m, p);
}

cudaError_t launch_advance(const AdvanceParams& a, cudaStream_t st) {
  return launch_chained(sc_advance_kernel, dim3(1), dim3(256), 0, st, a);
}

cudaError_t launch_export(const ExportParams& e, int ctas, cudaStream_t st) {
  const int items = (e.n_layers + 1) * e.B * ((e.L + kExportTokens - 1) / kExportTokens);
  return launch_chained(sc_export_kernel, dim3(std::max(1, std::min(items, ctas))),
                        dim3(kExportThreads), 0, st, e);
}

cudaError_t launch_gather(const GatherParams& g, cudaStream_t st) {
  const int nch = (g.L + kGatherTokens - 1) / kGatherTokens;
  if (g.gathered != nullptr) {
    // enough CTAs to keep the host link busy (about 2 MB in flight), few
    // enough that the items complete nearly in order, so that the first
    // sequences are in well before the last (measured on config 4 end to end:
    // 608 CTAs 0.489 ms, 152 0.484, 96 0.468, 64 0.469, 32 0.472)
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const int items = g.B * nch;
    return launch_chained(sc_gather_seq_kernel,
                          dim3(std::max(1, std::min(items, std::max(32, sms / 2)))),
                          dim3(kGatherThreads), 0, st, g);
  }
  dim3 grid(nch, g.B);
  return launch_chained(sc_gather_kernel, grid, dim3(kGatherThreads), 0, st, g);
}

}  // namespace sc
