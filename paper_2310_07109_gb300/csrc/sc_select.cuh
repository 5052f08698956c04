// sc_select.cuh -- the top-ratio keep rule on the device.
//
// The "top-k of the sequence length" family of Sec. "Pruning": a layer keeps
// k = ceil(rho n) of its n tokens (clamped to 1..n), the first token (always
// kept, as under the threshold rule) and the k-1 other tokens with the
// largest scores s_j, ties going to the lower current index.
//
// The cut is found by an MSB-first radix select with 8-bit digits over the
// block's candidates: scores are >= 0, so the order of their bit patterns as
// unsigned integers is the order of the scores.  One shared 256-bin histogram
// per digit, one warp to locate the digit that holds the (k-1)-th largest
// key, four digits in all; exact ties at the cut are ranked by index with
// warp ballots in index order.
#pragma once
#include <cstdint>

namespace sc {

// Kept tokens of the top-ratio rule for n current tokens and ratio rho:
// ceil(rho n) in double (exact for a float rho and n < 2^24), clamped to 1..n.
__device__ __forceinline__ int top_count(float rho, int n) {
  if (n <= 0) return 0;
  const double c = ceil(static_cast<double>(rho) * static_cast<double>(n));
  if (!(c >= 1.0)) return 1;   // also a NaN ratio
  return c >= static_cast<double>(n) ? n : static_cast<int>(c);
}

// Selection key of a candidate token (current index >= 1): its score's bit
// pattern plus one, so that every candidate has a key >= 1 and key 0 marks a
// non-candidate.  Scores are sums of probabilities (>= +0); a score that is
// not > 0 takes the lowest candidate key.
__device__ __forceinline__ uint32_t select_key(float s) {
  return s > 0.f ? __float_as_uint(s) + 1u : 1u;
}

struct SelectSmem {
  uint32_t hist[256];
  int sel[3];   // chosen digit, candidates still to take in it, candidates in it
};

// Block-wide cut of the top-ratio rule.  The calling threads (ids 0..kThreads-1
// among those that `sync` synchronises) each hold kItems keys: item u of
// thread t is token u * kThreads + t.  `want` = number of candidates to keep,
// 0 <= want <= (number of candidates).  On return (the same on every thread):
// a candidate with key > cut is kept, one with key == cut is kept when its
// rank among the keys equal to cut (in token order) is below `ties`, and
// eq = the number of candidates whose key equals cut.
template <int kThreads, int kItems, class Sync>
__device__ __forceinline__ void radix_cut(const uint32_t (&key)[kItems], int want, int m,
                                          SelectSmem& ss, int tid, Sync sync,
                                          uint32_t& cut, int& ties, int& eq) {
  if (want <= 0) {   // nothing beyond token 0
    cut = 0xffffffffu;
    ties = 0;
    eq = 0;
    return;
  }
  if (want >= m) {   // every candidate (keys >= 1 > 0)
    cut = 0u;
    ties = 0;
    eq = 0;
    return;
  }
  const int lane = tid & 31;
  uint32_t prefix = 0u, mask = 0u;
  int rem = want;
  int in_bin = 0;
#pragma unroll 1
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = tid; i < 256; i += kThreads) ss.hist[i] = 0u;
    sync();
#pragma unroll
    for (int u = 0; u < kItems; ++u)
      if (key[u] != 0u && (key[u] & mask) == prefix) atomicAdd(&ss.hist[(key[u] >> shift) & 255u], 1u);
    sync();
    if (tid < 32) {
      // lane l holds bins 255 - 8 l .. 248 - 8 l, largest first
      int c[8], tot = 0;
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        c[e] = static_cast<int>(ss.hist[255 - 8 * lane - e]);
        tot += c[e];
      }
      int incl = tot;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += y;
      }
      int cum = incl - tot;   // candidates in larger bins than this lane's
      if (cum < rem && rem <= incl) {
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          if (cum + c[e] >= rem) {
            ss.sel[0] = 255 - 8 * lane - e;
            ss.sel[1] = rem - cum;
            ss.sel[2] = c[e];
            break;
          }
          cum += c[e];
        }
      }
    }
    sync();
    const uint32_t digit = static_cast<uint32_t>(ss.sel[0]);
    rem = ss.sel[1];
    in_bin = ss.sel[2];
    prefix |= digit << shift;
    mask |= 255u << shift;
  }
  cut = prefix;
  ties = rem;
  eq = in_bin;
}

// Rank of the candidates equal to `cut` among themselves, in token order:
// flag[i] (one byte per token, i < n) is set here to 2 for the first `ties`
// of them and 1 for the others; the block reads it after the final sync.
// Only needed when eq > ties (an exact tie straddles the cut).
template <int kThreads, int kItems, class Sync>
__device__ __forceinline__ void rank_ties(const uint32_t (&key)[kItems], uint32_t cut, int ties,
                                          int n, uint8_t* flag, int tid, Sync sync) {
#pragma unroll
  for (int u = 0; u < kItems; ++u) {
    const int i = u * kThreads + tid;
    if (i < n) flag[i] = key[u] == cut ? 1 : 0;
  }
  sync();
  if (tid < 32) {
    const int lane = tid;
    int run = 0;
    for (int base = 0; base < n; base += 32) {
      const int i = base + lane;
      const bool f = i < n && flag[i] != 0;
      const uint32_t bal = __ballot_sync(0xffffffffu, f);
      if (f && run + __popc(bal & ((1u << lane) - 1u)) < ties) flag[i] = 2;
      run += __popc(bal);
    }
  }
  sync();
}

}  // namespace sc
