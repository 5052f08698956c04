// sc_internal.cuh -- parameter block shared by the host launcher and the
// kernels of the sparse-attention + token-pruning layer.
#pragma once

#include <cstdint>
#include <cuda.h>

#include "../../include/sparsecoder.h"

namespace sc {

constexpr int kHeadDim = 64;
constexpr int kTile = 128;         // rows (queries or keys) per tile
constexpr int kMaxBandTiles = 5;   // key (query) tiles touched by one 128-row tile, w <= 256
constexpr int kWideBandTiles = 9;  // ... with a wide window, 256 < w <= 512
constexpr int kPairWindow = 256;   // widest window of the paired rows layout on long sequences
constexpr int kMaxGlobal = 16;     // global tokens per sequence (one 16-wide MMA tile)
constexpr int kMaxLen = 4096;
constexpr int kMaxTiles = kMaxLen / kTile;
constexpr uint32_t kTileBytes = kTile * kHeadDim * 2;   // 16 KB bf16 tile
constexpr uint32_t kGTileBytes = kMaxGlobal * kHeadDim * 2;

// status word bits (workspace)
constexpr int kStatusTimeout = 1;
constexpr int kStatusInternal = 2;   // an invariant of the launch sequence did not hold

// Sequences with at most kTailMax current tokens run their remaining layers in
// the cluster kernel (one CTA per head); the per-layer kernels skip them.
constexpr int kTailMax = SC_TAIL_MAX_LEN;
constexpr int kTailMaxLayers = 64;
constexpr int kTailMaxHeads = 16;   // largest (non-portable) cluster

// log2(e) / sqrt(64): logits are kept in base-2 units, x = (q.k) * kLogitScale2.
// keep rules (the SC_KEEP_* values of the C interface)
constexpr int kKeepRelative = SC_KEEP_RELATIVE;
constexpr int kKeepAbsolute = SC_KEEP_ABSOLUTE;
constexpr int kKeepTopRatio = SC_KEEP_TOP_RATIO;

constexpr float kLogitScale2 = 0.125f * 1.4426950408889634f;

// TMA descriptors of Q, K, V (index 0, 1, 2) for both row sources: [0] the
// caller's tensors, [1] the compacted copies.  tile: 3-D [tokens][H][64] with a
// 128-token x 1-head box; row: 2-D [tokens*H][64] with a one-row box (gather4).
struct TensorMaps {
  CUtensorMap tile[2][3];
  CUtensorMap row[2][3];
};

struct LayerParams {
  int B, L, H, w;
  int T;                 // tiles per padded sequence = ceil(L / 128)
  // Where the current rows of sequence b live: when ident[b] != 0 (the current
  // tokens are original positions 0..n-1) row c is token (src_base + b*L + c)
  // of the "source" tensors; otherwise it is token (b*L + c) of the compacted
  // copies written by the gather kernel.
  long long src_base;    // token offset of this layer's [B][L] block in the source tensors
  const int32_t* ident;  // [B]
  const int32_t* len;    // [B] current lengths
  const int32_t* pos;    // [B][L] original positions of current tokens
  const int32_t* gcur;   // [B][kMaxGlobal] current indices of global tokens (increasing)
  const int32_t* ng;     // [B] number of global tokens present
  uint16_t* O;           // [B][L][H][64] bf16 out
  float* scores;         // [B][L] out
  int32_t* pos_out;      // [B][L] out
  int32_t* len_out;      // [B] out
  int32_t* gcur_out;     // [B][kMaxGlobal] out (next layer)
  int32_t* ng_out;       // [B] out
  int32_t* ident_out;    // [B] out (next layer)
  float alpha;           // the keep rule's value (alpha, theta or kept ratio)
  const float* theta;    // [B] absolute thresholds or nullptr (threshold rules)
  int keep_rule;         // kKeepRelative, kKeepAbsolute or kKeepTopRatio
  // workspace
  float* acc;            // [B][H][L] per-head column sums: band rows + global rows
  float* colpart;        // [B][H][L][band_slots] band-row column sums per query tile
                         //   (slot = query tile mod band_slots)
  int band_slots;        // kMaxBandTiles, or kWideBandTiles with wide
  int wide;              // rows kernel: one query tile per CTA (256 < w on long sequences)
  int band;              // the single-pass band kernel computes the rows (w <= 256)
  int sms;               // multiprocessors of the device (the band kernel's grid)
  float* gpart;          // [B][H][T][4][kMaxGlobal] column sums of global keys over far rows,
                         //   per (query tile, 32-row warp slice)
  float* gstat;          // [B][H][T][4][kMaxGlobal][2] (max, sum) of global rows per
                         //   (key tile, 32-key warp slice)
  float* og;             // [B][H][T2][kMaxGlobal][64] fp32 parts of the global rows'
                         //   outputs, one per key-tile pair (T2 = (T + 1) / 2)
  uint8_t* keep;         // [B][L]
  uint32_t* cnt_tile;    // [B][T]
  uint32_t* cnt_seq;     // [B]
  uint32_t* rows_done;   // [B][H]: rows CTAs of (sequence, head) whose results are visible
  uint32_t* cols_done;   // [B][H]: cols CTAs of (sequence, head) whose global-row parts are stored
  // nonzero: the gather kernel before this launch is still copying later
  // sequences' rows when it starts: sequence b's rows are complete once
  // gathered[b] reaches gather_target (the rows and cols kernels wait for it
  // instead of for the whole gather grid)
  const uint32_t* gathered;
  uint32_t gather_target;
  int32_t* kept_cur;     // [B][L] out, or nullptr: current index of each kept token, in order
  int* status;
  // test hook: when nonzero, the first MMA-issuing thread of every rows CTA
  // first waits at most this many nanoseconds on a barrier that nothing
  // completes, so that the bounded wait expires and the CTA aborts
  unsigned long long stall_ns;
  // hand-over to the cluster kernel: sequence b is skipped here once
  // tail_from[b] <= layer; the finalize of a layer sets tail_from[b] = layer + 1
  // when at most tail_max tokens survive.  tail_from == nullptr: no hand-over.
  int32_t* tail_from;    // [B]
  int layer;
  int tail_max;
  // nonzero: the source tensors are host memory, which the tensor maps never
  // read: every layer's rows are gathered (ident is never set)
  int no_ident;
  // Device-driven layer loop (a CUDA graph WHILE node): when dev_layer is set,
  // the layer is *dev_layer and the per-layer fields above hold their layer-0
  // values, advanced by these strides (gcur/ng/ident swap slots on odd layers;
  // alpha comes from alphas[layer]).
  const int* dev_layer;
  long long tok_stride;   // tokens of one layer in the source tensors (B * L)
  long long row_stride;   // entries of one layer in pos, pos_out, scores (B * L)
  long long o_stride;     // elements of one layer in O (B * L * H * 64)
  // O == nullptr: only the last layer's O is written, to O_last (when set)
  uint16_t* O_last;
  int n_layers;
  int len_stride;         // entries of one layer in len, len_out (B)
  float alphas[kTailMaxLayers];
};

// The per-layer fields of one launch, resolved (see layer_view in sc_kernels.cu).
struct LayerView {
  int layer;
  long long src_base;
  const int32_t* len;
  int32_t* len_out;
  const int32_t* pos;
  int32_t* pos_out;
  const int32_t* gcur;
  int32_t* gcur_out;
  const int32_t* ng;
  int32_t* ng_out;
  const int32_t* ident;
  int32_t* ident_out;
  uint16_t* O;
  float* scores;
  float alpha;
};

// Copies the rows of the kept tokens (at their original positions) of one
// layer's Q, K, V into compacted [B][L][H][64] buffers.
struct GatherParams {
  int B, L, H;
  long long src_base;          // token offset of the layer's [B][L] block in the sources
  const int32_t* len;          // [B]
  const int32_t* pos;          // [B][L]
  const int32_t* ident;        // [B]: sequences whose rows need no copy
  const uint16_t* src[3];      // Q, K, V sources [.., B, L, H, 64]
  uint16_t* dst[3];            // compacted Q, K, V [B][L][H][64]
  const int32_t* tail_from;    // [B] or nullptr: skip b when tail_from[b] <= layer
  int layer;                   // the layer whose rows are gathered
  // device-driven layer loop: the gathered layer is *dev_layer + 1, len/pos
  // above are those of layer 0 (advanced by the strides), ident alternates
  // between the two slots; nothing is gathered past the last layer
  const int* dev_layer;
  int n_layers;
  long long tok_stride, row_stride;
  int len_stride;
  const int32_t* ident_slot[2];
  // nonzero (sc_gather_seq_kernel, the layer given explicitly): the CTAs walk
  // the 8-token items sequence by sequence (grid stride) and raise
  // gathered[b] (release) once an item of sequence b is copied, so that the
  // next kernel can start on sequence b while later sequences are still being
  // copied (layer 0 of the host-buffer call, whose rows cross the host link);
  // their successors are launched only once the kernels before this one are
  // complete
  uint32_t* gathered;          // [B]
};

// One step of the device-driven layer loop: layer += 1, and the loop goes on
// while some sequence still runs through the per-layer kernels.
struct AdvanceParams {
  int B, n_layers;
  int* dev_layer;
  const int32_t* tail_from;
  unsigned long long cond;     // cudaGraphConditionalHandle of the WHILE node
};

struct PrepParams {
  int B, L;
  const uint8_t* pad_mask;   // [B][L] or nullptr (stack mode)
  const int32_t* pos_in;     // [B][L] given positions (layer mode) or nullptr
  const int32_t* len_in;     // [B] (layer mode)
  int32_t* pos_out;          // [B][L] (stack mode)
  int32_t* len_out;          // [B] (stack mode)
  int32_t* gcur;             // [B][kMaxGlobal]
  int32_t* ng;               // [B]
  int32_t* ident;            // [B]
  int32_t* tail_from;        // [B] (stack mode with the cluster kernel) or nullptr
  int tail_max;
  int* dev_layer;            // device-driven loop: set to 0 here, or nullptr
  unsigned long long cond;   // ... and its WHILE condition: some sequence has > tail_max tokens
  int has_cond;
  int no_ident;              // see LayerParams::no_ident
  int n_global;
  int global_pos[kMaxGlobal];
};

// Copies the results of a stack from the device to page-locked host memory:
// len[l][b] for every l <= n_layers, and for each (l, b) the first len[l][b]
// entries of pos (l <= n_layers), scores and O rows (l < n_layers).
struct ExportParams {
  int n_layers, B, L, H;
  const uint16_t* O;           // device [n_layers][B][L][H][64]
  const float* scores;         // device [n_layers][B][L]
  const int32_t* pos;          // device [n_layers + 1][B][L]
  const int32_t* len;          // device [n_layers + 1][B]
  uint16_t* hO;                // host (device-mapped addresses), same layouts; or nullptr:
  uint16_t* hO_last;           //   only the last layer's O rows, to hO_last [B][L][H][64]
  float* hscores;
  int32_t* hpos;
  int32_t* hlen;
  // part 0: every layer.  With the cluster kernel, part 1 copies the layers
  // l < tail_from[b], complete before that kernel, while it runs (the cluster
  // kernel writes the layers l >= tail_from[b] to the host buffers itself);
  // part 2, the layers l >= tail_from[b] from the device copies, is not used
  // by the host-buffer call.
  int part;
  const int32_t* tail_from;    // [B] (parts 1 and 2)
};

struct TailParams {
  int n_layers, B, L, H, w;
  const int32_t* tail_from;    // [B] first layer run here (>= n_layers: none)
  int32_t* pos;                // [n_layers + 1][B][L]
  int32_t* len;                // [n_layers + 1][B]
  uint16_t* O;                 // [n_layers][B][L][H][64], or nullptr: ...
  uint16_t* O_last;            // ... only the last layer's [B][L][H][64] (when set)
  float* scores;               // [n_layers][B][L]
  int* status;
  const uint16_t* src[3];      // Q, K, V [n_layers][B][L][H][64]
  // nonzero: src is host memory; the next layer's rows are not prefetched
  // (that would pull the rows of the tokens a layer prunes over the host link)
  int src_host;
  // host-buffer call: the results of the layers run here go straight to the
  // caller's page-locked buffers (device-mapped addresses, same layouts as
  // O / O_last / scores / pos / len): the entering layer's len and pos, then
  // each layer's O rows, scores, next pos and len; nullptr: device results
  // as above
  uint16_t* hO;
  uint16_t* hO_last;
  float* hscores;
  int32_t* hpos;
  int32_t* hlen;
  int n_global;
  int global_pos[kMaxGlobal];
  float alpha[kTailMaxLayers];   // the keep rule's value per layer
  int keep_rule;
};

// One GEMM of the encoder layer: out[(b, r)][n] = epi(sum_k A[row_a][k] W[n][k])
// for r < rows[b], row_a = b L + (a_idx ? a_idx[b L + r] : r); epi adds bias[n],
// then GELU (gelu != 0), then the bf16 residual res[row][n] (row = b L +
// (res_idx ? res_idx[b L + r] : r)).  N % 128 == 0, K % 64 == 0; tiles of 128 rows
// by bn columns.
struct GemmParams {
  CUtensorMap map_a;               // 2-D [B L][K] bf16, box 64 x 1 (four-row gathers)
  CUtensorMap map_at;              // the same matrix, box 64 x 128 (consecutive rows)
  CUtensorMap map_w;               // 2-D [N][K] bf16, box 64 x wbox
  int B, L, N, K;
  int bn;                          // output columns per tile: 256, 192 or 128 (the width
                                   // that fills the SMs' rounds of tiles best)
  int wbox;                        // W rows per copy: min(bn, N)
  const int32_t* rows;             // [B] rows per sequence, or nullptr (L)
  const int32_t* a_idx;            // [B][L] A row of output row (b, r), or nullptr
  const float* bias;               // [N] or nullptr
  int gelu;
  const uint16_t* res;             // bf16 [B L][N] or nullptr
  const int32_t* res_idx;          // [B][L] residual row of output row (b, r), or nullptr
  void* out;                       // [B L][N], bf16 or fp32 (out_f32)
  int out_f32;
  int out_split;                   // > 0: column block j of width out_split goes to outs[j]
  void* outs[3];
  int* status;
};

// Layer norm over D features of the rows (b, r), r < rows[b]: fp32 in, bf16 out.
// Rows of a bf16 [B L][D] matrix gathered into consecutive rows:
// dst[b L + r] = src[b L + idx[b L + r]] for r < rows[b].
struct RowGatherParams {
  int B, L, D;
  const int32_t* rows;             // [B]
  const int32_t* idx;              // [B][L]
  const uint16_t* src;
  uint16_t* dst;
};

struct LayerNormParams {
  int B, L, D;
  const int32_t* rows;
  const float* in;
  const float* gamma;
  const float* beta;
  float eps;
  uint16_t* out;
  int vec;   // set by the launcher: D % 128 == 0 and aligned rows (4 features per access)
};

}  // namespace sc
