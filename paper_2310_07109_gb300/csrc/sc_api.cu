// sc_api.cu -- the C ABI declared in include/sparsecoder.h: argument checks,
// workspace layout, TMA descriptors and the launch sequence of one layer or
// of the pruned layer stack.  All launches go to the caller's stream; nothing
// here synchronises the host except sc_workspace_status().
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cmath>
#include <cstdint>
#include <cstdio>
#include <atomic>
#include <cstring>
#include <functional>
#include <mutex>

#include "../../include/sparsecoder.h"
#include "sc_internal.cuh"

namespace sc {
cudaError_t launch_prep(const PrepParams& pp, cudaStream_t st);
cudaError_t configure_kernels();
cudaError_t launch_rows(const TensorMaps& m, const LayerParams& p, cudaStream_t st);
cudaError_t launch_cols(const TensorMaps& m, const LayerParams& p, cudaStream_t st);
cudaError_t launch_gather(const GatherParams& g, cudaStream_t st);
cudaError_t launch_export(const ExportParams& e, int ctas, cudaStream_t st);
cudaError_t launch_advance(const AdvanceParams& a, cudaStream_t st);
cudaError_t configure_tail();
cudaError_t tail_max_clusters(int H, int* out);
cudaError_t launch_tail(const TailParams& p, cudaStream_t st);
cudaError_t configure_encoder();
cudaError_t launch_gemm(const GemmParams& p, cudaStream_t st);
cudaError_t launch_layernorm(const LayerNormParams& p, cudaStream_t st);
cudaError_t launch_row_gather(const RowGatherParams& p, cudaStream_t st);
}  // namespace sc

namespace {

using namespace sc;

constexpr size_t kAlign = 256;

// Detail of the most recent failure on this thread (sc_last_error()).
thread_local char g_last_error[256] = "";

// Test hook of the failure path (sc_debug_stall_waits): nanoseconds that every
// rows CTA waits on a barrier that nothing completes; 0 = off.
std::atomic<unsigned long long> g_stall_ns{0};

// Which rows kernel computes the per-layer attention for windows up to 256
// (sc_select_rows_kernel): SC_ROWS_SINGLE_PASS or SC_ROWS_TWO_PASS.
std::atomic<int> g_rows_kernel{SC_ROWS_TWO_PASS};

// Multiprocessors of the current device (cached per device; 0 if unknown).
int device_sms() {
  static std::atomic<int> cache[256];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 256) {
    cudaGetLastError();
    return 0;
  }
  int v = cache[dev].load(std::memory_order_relaxed);
  if (v == 0) {
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
      cudaGetLastError();
      v = 0;
    }
    cache[dev].store(v, std::memory_order_relaxed);
  }
  return v;
}

int fail(int code, const char* what, const char* detail) {
  snprintf(g_last_error, sizeof g_last_error, "%s: %s", what, detail ? detail : "");
  return code;
}

int fail_cuda(const char* what, cudaError_t e) {
  return fail(SC_ERR_CUDA, what, cudaGetErrorString(e));
}

size_t align_up(size_t x) { return (x + kAlign - 1) & ~(kAlign - 1); }

struct WsLayout {
  size_t status, acc, colpart, gpart, gstat, og, keep, cnt_tile, cnt_seq, rows_done, cols_done,
      gathered, gcur, ng,
      ident,
      tail_from,
      loop_layer, qkv, total;
};

bool ws_layout(int B, int L, int H, WsLayout* w) {
  if (B < 1 || L < 1 || H < 1 || L > kMaxLen) return false;
  const size_t T = (L + kTile - 1) / kTile;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align_up(off + bytes);
    return at;
  };
  w->status = take(kAlign);
  w->acc = take(sizeof(float) * B * H * (size_t)L);
  w->colpart = take(sizeof(float) * B * H * (size_t)L * kWideBandTiles);
  w->gpart = take(sizeof(float) * B * H * T * 4 * kMaxGlobal);
  w->gstat = take(sizeof(float) * B * H * T * 4 * kMaxGlobal * 2);
  w->og = take(sizeof(float) * B * H * ((T + 1) / 2) * kMaxGlobal * kHeadDim);
  w->keep = take(sizeof(uint8_t) * B * (size_t)L);
  w->cnt_tile = take(sizeof(uint32_t) * B * T);
  w->cnt_seq = take(sizeof(uint32_t) * B);
  w->rows_done = take(sizeof(uint32_t) * B * H);
  w->cols_done = take(sizeof(uint32_t) * B * H);
  w->gathered = take(sizeof(uint32_t) * B);
  w->gcur = take(sizeof(int32_t) * 2 * B * kMaxGlobal);
  w->ng = take(sizeof(int32_t) * 2 * B);
  w->ident = take(sizeof(int32_t) * 2 * B);
  w->tail_from = take(sizeof(int32_t) * B);
  w->loop_layer = take(sizeof(int32_t));
  // compacted Q, K, V of the current layer (rows of the surviving tokens)
  w->qkv = take(sizeof(uint16_t) * 3 * B * (size_t)L * H * kHeadDim);
  w->total = off;
  return true;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

PFN_cuTensorMapEncodeTiled_v12000 get_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    cudaDriverEntryPointQueryResult q;
    void* ptr = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// Tile view: 3-D [tokens][H][64] of a bf16 tensor laid out (.., token, head,
// 64); one TMA box is 128 consecutive tokens of one head (16 KB).
bool encode_tiles(CUtensorMap* m, const void* base, long long tokens, int H) {
  auto enc = get_encoder();
  if (!enc) return fail(SC_ERR_CUDA, "tensor-map encoder", "cuTensorMapEncodeTiled unavailable"), false;
  cuuint64_t gdim[3] = {static_cast<cuuint64_t>(kHeadDim), static_cast<cuuint64_t>(H),
                        static_cast<cuuint64_t>(tokens)};
  cuuint64_t gstride[2] = {static_cast<cuuint64_t>(kHeadDim * 2),
                           static_cast<cuuint64_t>(kHeadDim * 2) * H};
  cuuint32_t box[3] = {static_cast<cuuint32_t>(kHeadDim), 1, static_cast<cuuint32_t>(kTile)};
  cuuint32_t estride[3] = {1, 1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), gdim, gstride,
                   box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    char d[64];
    snprintf(d, sizeof d, "CUresult %d", static_cast<int>(r));
    fail(SC_ERR_CUDA, "encode 3-D tile map", d);
  }
  return r == CUDA_SUCCESS;
}

// Row view: 2-D [tokens * H][64]; one TMA box is a single 128-byte row,
// gathered four at a time (the global tokens).
bool encode_rows(CUtensorMap* m, const void* base, long long rows) {
  auto enc = get_encoder();
  if (!enc) return fail(SC_ERR_CUDA, "tensor-map encoder", "cuTensorMapEncodeTiled unavailable"), false;
  cuuint64_t gdim[2] = {static_cast<cuuint64_t>(kHeadDim), static_cast<cuuint64_t>(rows)};
  cuuint64_t gstride[1] = {static_cast<cuuint64_t>(kHeadDim * 2)};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(kHeadDim), 1};
  cuuint32_t estride[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), gdim, gstride,
                   box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    char d[64];
    snprintf(d, sizeof d, "CUresult %d", static_cast<int>(r));
    fail(SC_ERR_CUDA, "encode 2-D row map", d);
  }
  return r == CUDA_SUCCESS;
}

// Plain 2-D view [rows][cols] of a bf16 matrix (row stride cols), 128-byte
// swizzle; one TMA box is 64 columns x box_rows rows.
bool encode_2d(CUtensorMap* m, const void* base, long long rows, int cols, int box_rows) {
  auto enc = get_encoder();
  if (!enc) return fail(SC_ERR_CUDA, "tensor-map encoder", "cuTensorMapEncodeTiled unavailable"), false;
  cuuint64_t gdim[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows)};
  cuuint64_t gstride[1] = {static_cast<cuuint64_t>(cols) * 2};
  cuuint32_t box[2] = {64u, static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estride[2] = {1, 1};
  CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), gdim, gstride,
                   box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) {
    char d[64];
    snprintf(d, sizeof d, "CUresult %d", static_cast<int>(r));
    fail(SC_ERR_CUDA, "encode 2-D matrix map", d);
  }
  return r == CUDA_SUCCESS;
}

// Descriptors for the caller's Q, K, V (source 0, `tokens` tokens) and the
// compacted copies in the workspace (source 1, B * L tokens).
bool encode_maps(TensorMaps* m, const uint16_t* const src[3], long long tokens, uint16_t* const cmp[3],
                 long long cmp_tokens, int H) {
  for (int t = 0; t < 3; ++t) {
    if (!encode_tiles(&m->tile[0][t], src[t], tokens, H) ||
        !encode_rows(&m->row[0][t], src[t], tokens * H) ||
        !encode_tiles(&m->tile[1][t], cmp[t], cmp_tokens, H) ||
        !encode_rows(&m->row[1][t], cmp[t], cmp_tokens * H))
      return false;
  }
  return true;
}

cudaStream_t capture_side_stream();

int ensure_configured() {
  static std::mutex mu;
  static bool done[256] = {false};
  int dev = 0;
  const cudaError_t ge = cudaGetDevice(&dev);
  if (ge != cudaSuccess) return fail_cuda("cudaGetDevice", ge);
  if (dev < 0 || dev >= 256) return fail(SC_ERR_CUDA, "cudaGetDevice", "device index out of range");
  std::lock_guard<std::mutex> lock(mu);
  if (!done[dev]) {
    cudaError_t e = configure_kernels();
    if (e == cudaSuccess) e = configure_tail();
    if (e == cudaSuccess) e = configure_encoder();
    if (e != cudaSuccess) return fail_cuda("kernel attributes", e);
    done[dev] = true;
  }
  capture_side_stream();   // made outside any capture when possible
  return SC_OK;
}

// A stream of this library per device, used only to record the body of the
// layer loop into a graph under construction (nullptr if it cannot be made).
cudaStream_t capture_side_stream() {
  static std::mutex mu;
  static cudaStream_t side[256] = {nullptr};
  static bool tried[256] = {false};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 256) {
    cudaGetLastError();
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (!tried[dev]) {
    tried[dev] = true;
    if (cudaStreamCreateWithFlags(&side[dev], cudaStreamNonBlocking) != cudaSuccess) {
      cudaGetLastError();
      side[dev] = nullptr;
    }
  }
  return side[dev];
}

// Whether the cluster kernel can run with clusters of H CTAs on the current
// device (cached per device and H; call after ensure_configured()).
int tail_available(int H, bool* ok) {
  static std::mutex mu;
  static signed char state[256][kTailMaxHeads + 1];   // 0 unknown, 1 yes, -1 no
  *ok = false;
  if (H < 1 || H > kTailMaxHeads) return SC_OK;
  int dev = 0;
  const cudaError_t ge = cudaGetDevice(&dev);
  if (ge != cudaSuccess) return fail_cuda("cudaGetDevice", ge);
  if (dev < 0 || dev >= 256) return fail(SC_ERR_CUDA, "cudaGetDevice", "device index out of range");
  std::lock_guard<std::mutex> lock(mu);
  if (state[dev][H] == 0) {
    int clusters = 0;
    const cudaError_t e = tail_max_clusters(H, &clusters);
    if (e != cudaSuccess) {
      cudaGetLastError();   // an unsupported shape is not an error of the call
      clusters = 0;
    }
    state[dev][H] = clusters > 0 ? 1 : -1;
  }
  *ok = state[dev][H] > 0;
  return SC_OK;
}

int check_common(int B, int L, int H, int w, const int32_t* gpos, int ngl) {
  if (B < 1 || L < 1 || H < 1 || w < 0 || ngl < 0) return SC_ERR_INVALID_ARG;
  if (L > SC_MAX_LEN) return SC_ERR_UNSUPPORTED;
  if (ngl > SC_MAX_GLOBAL) return SC_ERR_UNSUPPORTED;
  if (ngl > 0 && gpos == nullptr) return SC_ERR_INVALID_ARG;
  for (int g = 0; g < ngl; ++g) {
    if (gpos[g] < 0 || gpos[g] >= L) return SC_ERR_INVALID_ARG;
    if (g > 0 && gpos[g] <= gpos[g - 1]) return SC_ERR_INVALID_ARG;
  }
  // one 128-row tile must reach at most nine 128-key tiles
  if (L > kMaxBandTiles * kTile && w > SC_MAX_WINDOW) return SC_ERR_UNSUPPORTED;
  if (static_cast<long long>(B) * L * H > (1ll << 30)) return SC_ERR_UNSUPPORTED;
  return SC_OK;
}

// The keep rule and its per-layer values (one value for a layer call): the
// top-ratio rule takes no per-sequence thresholds and needs finite ratios.
int check_keep(int rule, const float* values, int count, const float* theta) {
  if (rule != SC_KEEP_RELATIVE && rule != SC_KEEP_ABSOLUTE && rule != SC_KEEP_TOP_RATIO)
    return fail(SC_ERR_INVALID_ARG, "keep_rule", "not an sc_keep_rule");
  if (rule == SC_KEEP_TOP_RATIO) {
    if (theta) return fail(SC_ERR_INVALID_ARG, "theta", "the top-ratio rule takes no thresholds");
    for (int l = 0; l < count; ++l)
      if (!std::isfinite(values[l])) return fail(SC_ERR_INVALID_ARG, "alpha", "ratio not finite");
  }
  return SC_OK;
}

void fill_workspace(LayerParams* p, char* ws, const WsLayout& lay, int slot) {
  p->status = reinterpret_cast<int*>(ws + lay.status);
  p->acc = reinterpret_cast<float*>(ws + lay.acc);
  p->colpart = reinterpret_cast<float*>(ws + lay.colpart);
  p->gpart = reinterpret_cast<float*>(ws + lay.gpart);
  p->gstat = reinterpret_cast<float*>(ws + lay.gstat);
  p->og = reinterpret_cast<float*>(ws + lay.og);
  p->keep = reinterpret_cast<uint8_t*>(ws + lay.keep);
  p->cnt_tile = reinterpret_cast<uint32_t*>(ws + lay.cnt_tile);
  p->cnt_seq = reinterpret_cast<uint32_t*>(ws + lay.cnt_seq);
  p->rows_done = reinterpret_cast<uint32_t*>(ws + lay.rows_done);
  p->cols_done = reinterpret_cast<uint32_t*>(ws + lay.cols_done);
  p->stall_ns = g_stall_ns.load(std::memory_order_relaxed);
  int32_t* gcur = reinterpret_cast<int32_t*>(ws + lay.gcur);
  int32_t* ng = reinterpret_cast<int32_t*>(ws + lay.ng);
  int32_t* ident = reinterpret_cast<int32_t*>(ws + lay.ident);
  p->gcur = gcur + slot * p->B * kMaxGlobal;
  p->gcur_out = gcur + (1 - slot) * p->B * kMaxGlobal;
  p->ng = ng + slot * p->B;
  p->ng_out = ng + (1 - slot) * p->B;
  p->ident = ident + slot * p->B;
  p->ident_out = ident + (1 - slot) * p->B;
  // rows kernel layout: pairs of query tiles, or single tiles when a tile's
  // band reaches more than five key tiles
  p->wide = (p->w > kPairWindow && p->T > kMaxBandTiles) ? 1 : 0;
  p->band_slots = p->wide ? kWideBandTiles : kMaxBandTiles;
  p->sms = device_sms();
  p->band = (!p->wide && p->sms > 0 &&
             g_rows_kernel.load(std::memory_order_relaxed) == SC_ROWS_SINGLE_PASS) ? 1 : 0;
}

void compacted_qkv(char* ws, const WsLayout& lay, int B, int L, int H, uint16_t* out[3]) {
  const size_t per = static_cast<size_t>(B) * L * H * kHeadDim;
  uint16_t* base = reinterpret_cast<uint16_t*>(ws + lay.qkv);
  for (int t = 0; t < 3; ++t) out[t] = base + t * per;
}

int reset_counters(char* ws, const WsLayout& lay, cudaStream_t st) {
  // the counters reset themselves after each layer; clearing them per call
  // keeps a call independent of any earlier call that was cut short
  const cudaError_t e = cudaMemsetAsync(ws + lay.cnt_tile, 0, lay.gcur - lay.cnt_tile, st);
  if (e != cudaSuccess) return fail_cuda("counter reset", e);
  return SC_OK;
}

}  // namespace

extern "C" {

size_t sc_workspace_size(int B, int L, int H) {
  WsLayout lay;
  if (!ws_layout(B, L, H, &lay)) return 0;
  return lay.total;
}

const char* sc_last_error(void) { return g_last_error; }

const char* sc_status_string(int status) {
  switch (status) {
    case SC_OK: return "SC_OK";
    case SC_ERR_INVALID_ARG: return "SC_ERR_INVALID_ARG: invalid argument";
    case SC_ERR_UNSUPPORTED: return "SC_ERR_UNSUPPORTED: size or option outside the supported range";
    case SC_ERR_CUDA: return "SC_ERR_CUDA: a CUDA call failed";
    case SC_ERR_TIMEOUT: return "SC_ERR_TIMEOUT: a bounded device-side wait expired";
    case SC_ERR_WORKSPACE: return "SC_ERR_WORKSPACE: workspace missing, too small or misaligned";
    default: return "unknown sparsecoder status";
  }
}

namespace {
int layer_forward_impl(const sc_layer_args* a, void* workspace, size_t ws_bytes, void* stream,
                       int32_t* kept_cur);
}  // namespace

int sc_layer_forward(const sc_layer_args* a, void* workspace, size_t ws_bytes, void* stream) {
  return layer_forward_impl(a, workspace, ws_bytes, stream, nullptr);
}

namespace {
// One layer; kept_cur (device [B][L] or nullptr) receives the current index of
// each kept token, in order.
int layer_forward_impl(const sc_layer_args* a, void* workspace, size_t ws_bytes, void* stream,
                       int32_t* kept_cur) {
  if (!a) return SC_ERR_INVALID_ARG;
  int rc = check_common(a->B, a->L, a->H, a->w, a->global_pos, a->n_global);
  if (rc != SC_OK) return rc;
  if (!a->Q || !a->K || !a->V || !a->len || !a->pos || !a->O || !a->scores || !a->pos_out ||
      !a->len_out)
    return SC_ERR_INVALID_ARG;
  if (!aligned16(a->Q) || !aligned16(a->K) || !aligned16(a->V) || !aligned16(a->O))
    return SC_ERR_INVALID_ARG;
  if (a->pos_out == a->pos || a->len_out == a->len) return SC_ERR_INVALID_ARG;
  if ((rc = check_keep(a->keep_rule, &a->alpha, 1, a->theta)) != SC_OK) return rc;
  WsLayout lay;
  ws_layout(a->B, a->L, a->H, &lay);
  if (!workspace || ws_bytes < lay.total || (reinterpret_cast<uintptr_t>(workspace) % kAlign))
    return SC_ERR_WORKSPACE;
  if ((rc = ensure_configured()) != SC_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  char* ws = static_cast<char*>(workspace);

  TensorMaps maps;
  uint16_t* cmp[3];
  compacted_qkv(ws, lay, a->B, a->L, a->H, cmp);
  const uint16_t* src[3] = {a->Q, a->K, a->V};
  const long long tokens = static_cast<long long>(a->B) * a->L;
  if (!encode_maps(&maps, src, tokens, cmp, tokens, a->H)) return SC_ERR_CUDA;
  if ((rc = reset_counters(ws, lay, st)) != SC_OK) return rc;

  LayerParams p{};
  p.B = a->B; p.L = a->L; p.H = a->H; p.w = a->w;
  p.T = (a->L + kTile - 1) / kTile;
  p.src_base = 0;
  p.len = a->len;
  p.pos = a->pos;
  p.O = a->O;
  p.scores = a->scores;
  p.pos_out = a->pos_out;
  p.len_out = a->len_out;
  p.alpha = a->alpha;
  p.theta = a->theta;
  p.keep_rule = a->keep_rule;
  fill_workspace(&p, ws, lay, 0);
  p.kept_cur = kept_cur;

  PrepParams pp{};
  pp.B = a->B; pp.L = a->L;
  pp.pos_in = a->pos;
  pp.len_in = a->len;
  pp.gcur = const_cast<int32_t*>(p.gcur);
  pp.ng = const_cast<int32_t*>(p.ng);
  pp.ident = const_cast<int32_t*>(p.ident);
  pp.n_global = a->n_global;
  for (int g = 0; g < a->n_global; ++g) pp.global_pos[g] = a->global_pos[g];
  cudaError_t e;
  if ((e = launch_prep(pp, st)) != cudaSuccess) return fail_cuda("launch prep kernel", e);
  if ((e = launch_rows(maps, p, st)) != cudaSuccess) return fail_cuda("launch rows kernel", e);
  if ((e = launch_cols(maps, p, st)) != cudaSuccess) return fail_cuda("launch cols kernel", e);
  return SC_OK;
}
}  // namespace

// Which kernels a stack call launches: sequences with at most kTailMax tokens
// left finish in the cluster kernel (when it can run with clusters of H CTAs);
// with L <= kTailMax every sequence starts there and no per-layer kernel runs.
static int stack_plan(const sc_stack_args* a, bool* use_tail, bool* per_layer) {
  const int n_layers = a->n_layers, L = a->L, H = a->H;
  bool ok = false;
  if (!(a->flags & SC_STACK_NO_TAIL)) {
    const int rc = tail_available(H, &ok);
    if (rc != SC_OK) return rc;
  }
  *use_tail = ok && n_layers <= kTailMaxLayers;
  *per_layer = !*use_tail || L > kTailMax;
  return SC_OK;
}

// The caller's page-locked result buffers of a host-buffer call (device-mapped
// addresses): the cluster kernel writes its layers' results there directly.
struct HostResults {
  uint16_t* O;
  uint16_t* O_last;
  float* scores;
  int32_t* pos;
  int32_t* len;
};

// host_io: Q, K, V (and pad_mask) are device-mapped addresses of host memory,
// which only the gather and cluster kernels read (plain loads): the tensor
// maps of the "source" slot are pointed at the compacted copies and never
// selected, and every layer's rows are gathered; hres (host_io only): where
// the cluster kernel puts its results.
// The argument checks of a stack call (nothing is enqueued).
static int stack_check(const sc_stack_args* a, void* workspace, size_t ws_bytes) {
  if (!a) return SC_ERR_INVALID_ARG;
  if (a->n_layers < 1 || (a->flags & ~(SC_STACK_NO_TAIL | SC_STACK_PLAIN_LAUNCHES)))
    return SC_ERR_INVALID_ARG;
  int rc = check_common(a->B, a->L, a->H, a->w, a->global_pos, a->n_global);
  if (rc != SC_OK) return rc;
  if (!a->Q || !a->K || !a->V || !a->alpha || !a->scores || !a->pos || !a->len)
    return SC_ERR_INVALID_ARG;
  if ((rc = check_keep(a->keep_rule, a->alpha, a->n_layers, nullptr)) != SC_OK) return rc;
  if (!aligned16(a->Q) || !aligned16(a->K) || !aligned16(a->V) || !aligned16(a->O) ||
      !aligned16(a->O_last))
    return SC_ERR_INVALID_ARG;
  const long long rows = static_cast<long long>(a->n_layers) * a->B * a->L * a->H;
  if (rows > (1ll << 31) - 1) return SC_ERR_UNSUPPORTED;
  WsLayout lay;
  ws_layout(a->B, a->L, a->H, &lay);
  if (!workspace || ws_bytes < lay.total || (reinterpret_cast<uintptr_t>(workspace) % kAlign))
    return SC_ERR_WORKSPACE;
  return ensure_configured();
}

static int stack_forward_impl(const sc_stack_args* a, void* workspace, size_t ws_bytes,
                              void* stream, void** events, int n_events, bool host_io = false,
                              const HostResults* hres = nullptr) {
  int rc = stack_check(a, workspace, ws_bytes);
  if (rc != SC_OK) return rc;
  // the O of every layer, or (O == NULL) only the last layer's, to O_last
  uint16_t* const o_last = a->O != nullptr ? nullptr : a->O_last;
  WsLayout lay;
  ws_layout(a->B, a->L, a->H, &lay);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  char* ws = static_cast<char*>(workspace);

  TensorMaps maps;
  uint16_t* cmp[3];
  compacted_qkv(ws, lay, a->B, a->L, a->H, cmp);
  const uint16_t* src[3] = {a->Q, a->K, a->V};
  const long long BLt = static_cast<long long>(a->B) * a->L;
  const uint16_t* map_src[3] = {host_io ? cmp[0] : src[0], host_io ? cmp[1] : src[1],
                                host_io ? cmp[2] : src[2]};
  if (!encode_maps(&maps, map_src, host_io ? BLt : a->n_layers * BLt, cmp, BLt, a->H))
    return SC_ERR_CUDA;
  if ((rc = reset_counters(ws, lay, st)) != SC_OK) return rc;

  const size_t BL = static_cast<size_t>(a->B) * a->L;
  bool use_tail = false, per_layer = true;
  if ((rc = stack_plan(a, &use_tail, &per_layer)) != SC_OK) return rc;
  int32_t* tail_from = use_tail ? reinterpret_cast<int32_t*>(ws + lay.tail_from) : nullptr;

  LayerParams p{};
  p.B = a->B; p.L = a->L; p.H = a->H; p.w = a->w;
  p.T = (a->L + kTile - 1) / kTile;
  p.theta = nullptr;
  p.keep_rule = a->keep_rule;
  p.tail_from = tail_from;
  p.tail_max = use_tail ? kTailMax : 0;
  p.no_ident = host_io ? 1 : 0;
  p.n_layers = a->n_layers;
  fill_workspace(&p, ws, lay, 0);

  PrepParams pp{};
  pp.B = a->B; pp.L = a->L;
  pp.pad_mask = a->pad_mask;
  pp.pos_out = a->pos;
  pp.len_out = a->len;
  pp.gcur = const_cast<int32_t*>(p.gcur);
  pp.ng = const_cast<int32_t*>(p.ng);
  pp.ident = const_cast<int32_t*>(p.ident);
  pp.tail_from = tail_from;
  pp.tail_max = p.tail_max;
  pp.no_ident = p.no_ident;
  pp.n_global = a->n_global;
  for (int g = 0; g < a->n_global; ++g) pp.global_pos[g] = a->global_pos[g];
  auto mark = [&](int k) {
    return events == nullptr || events[k] == nullptr ||
           cudaEventRecord(static_cast<cudaEvent_t>(events[k]), st) == cudaSuccess;
  };
  cudaError_t e;

  // While the call is captured into a CUDA graph, the per-layer kernels run
  // in a WHILE node whose condition the device sets ("some sequence still has
  // more than kTailMax tokens"), with the layer index in device memory: layers
  // that every sequence has left cost no launch.  Uncaptured calls here (plain
  // launches, the profiled call) launch every layer's kernels, which then skip
  // the sequences of the cluster kernel; other eager calls reach this point
  // while the library records them into a graph of its own.
  bool dev_loop = false;
  cudaGraphConditionalHandle cond = 0;
  cudaStream_t side = nullptr;
  if (use_tail && per_layer && events == nullptr) {
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st, &cap) != cudaSuccess) {
      cudaGetLastError();
      cap = cudaStreamCaptureStatusNone;
    }
    if (cap == cudaStreamCaptureStatusActive) side = capture_side_stream();
    if (side != nullptr) {
      cudaGraph_t g = nullptr;
      cudaStreamCaptureStatus cs;
      if ((e = cudaStreamGetCaptureInfo(st, &cs, nullptr, &g)) != cudaSuccess)
        return fail_cuda("stream capture info", e);
      if ((e = cudaGraphConditionalHandleCreate(&cond, g, 0, cudaGraphCondAssignDefault)) !=
          cudaSuccess)
        return fail_cuda("conditional handle", e);
      dev_loop = true;
    }
  }
  int* loop_layer = reinterpret_cast<int*>(ws + lay.loop_layer);
  if (dev_loop) {
    pp.dev_layer = loop_layer;
    pp.cond = cond;
    pp.has_cond = 1;
  }

  if (!mark(0)) return fail(SC_ERR_CUDA, "event record", "");
  if ((e = launch_prep(pp, st)) != cudaSuccess) return fail_cuda("launch prep kernel", e);
  if (!mark(1)) return fail(SC_ERR_CUDA, "event record", "");
  // layer 0 reads the caller's rows in place when no padding was removed; the
  // gather kernel copies the survivors' rows for every later layer
  GatherParams gp{};
  gp.B = a->B; gp.L = a->L; gp.H = a->H;
  gp.tail_from = tail_from;
  for (int t = 0; t < 3; ++t) {
    gp.src[t] = src[t];
    gp.dst[t] = cmp[t];
  }
  // Host buffers: layer 0's rows cross the host link; the gather walks them
  // sequence by sequence and counts what it has copied, and layer 0's rows and
  // cols kernels start on a sequence as soon as its rows are in.
  uint32_t* const gathered = host_io ? reinterpret_cast<uint32_t*>(ws + lay.gathered) : nullptr;
  const uint32_t gather_target = static_cast<uint32_t>((a->L + 7) / 8);
  if (dev_loop) {
    if (a->pad_mask != nullptr || host_io) {
      // padding removal may have moved rows: compact layer 0 as well
      gp.src_base = 0;
      gp.layer = 0;
      gp.len = a->len;
      gp.pos = a->pos;
      gp.ident = p.ident;
      gp.gathered = gathered;
      if ((e = launch_gather(gp, st)) != cudaSuccess) return fail_cuda("launch gather kernel", e);
      gp.gathered = nullptr;
    }
    LayerParams pd = p;   // workspace slot 0: layer 0's ping-pong buffers
    pd.dev_layer = loop_layer;
    pd.layer = 0;
    pd.src_base = 0;
    pd.len = a->len;
    pd.len_out = a->len + a->B;
    pd.pos = a->pos;
    pd.pos_out = a->pos + BL;
    pd.O = a->O;
    pd.O_last = o_last;
    pd.scores = a->scores;
    pd.alpha = a->alpha[0];
    pd.tok_stride = BLt;
    pd.row_stride = static_cast<long long>(BL);
    pd.o_stride = static_cast<long long>(BL) * a->H * kHeadDim;
    pd.len_stride = a->B;
    for (int l = 0; l < a->n_layers; ++l) pd.alphas[l] = a->alpha[l];
    GatherParams gd = gp;
    gd.dev_layer = loop_layer;
    gd.n_layers = a->n_layers;
    gd.tok_stride = BLt;
    gd.row_stride = static_cast<long long>(BL);
    gd.len_stride = a->B;
    gd.len = a->len;
    gd.pos = a->pos;
    gd.ident_slot[0] = p.ident;
    gd.ident_slot[1] = p.ident_out;
    AdvanceParams ad{};
    ad.B = a->B;
    ad.n_layers = a->n_layers;
    ad.dev_layer = loop_layer;
    ad.tail_from = tail_from;
    ad.cond = cond;

    // layer 0 ahead of the loop (chained to the kernels before it), the loop
    // from layer 1 on: the advance kernel sets the loop's condition
    {
      LayerParams p0 = pd;
      p0.gathered = gathered;
      p0.gather_target = gather_target;
      cudaError_t le0 = launch_rows(maps, p0, st);
      if (le0 == cudaSuccess) le0 = launch_cols(maps, p0, st);
      if (le0 == cudaSuccess) le0 = launch_gather(gd, st);
      if (le0 == cudaSuccess) le0 = launch_advance(ad, st);
      if (le0 != cudaSuccess) return fail_cuda("launch layer 0", le0);
    }
    cudaGraph_t g = nullptr;
    const cudaGraphNode_t* deps = nullptr;
    size_t ndeps = 0;
    cudaStreamCaptureStatus cs;
    if ((e = cudaStreamGetCaptureInfo(st, &cs, nullptr, &g, &deps, nullptr, &ndeps)) != cudaSuccess)
      return fail_cuda("stream capture info", e);
    cudaGraphNodeParams cp = {};
    cp.type = cudaGraphNodeTypeConditional;
    cp.conditional.handle = cond;
    cp.conditional.type = cudaGraphCondTypeWhile;
    cp.conditional.size = 1;
    cudaGraphNode_t node;
    if ((e = cudaGraphAddNode(&node, g, deps, nullptr, ndeps, &cp)) != cudaSuccess)
      return fail_cuda("add WHILE node", e);
    if ((e = cudaStreamBeginCaptureToGraph(side, cp.conditional.phGraph_out[0], nullptr, nullptr, 0,
                                           cudaStreamCaptureModeRelaxed)) != cudaSuccess)
      return fail_cuda("capture layer loop body", e);
    cudaError_t le = launch_rows(maps, pd, side);
    if (le == cudaSuccess) le = launch_cols(maps, pd, side);
    if (le == cudaSuccess) le = launch_gather(gd, side);
    if (le == cudaSuccess) le = launch_advance(ad, side);
    cudaGraph_t body = nullptr;
    e = cudaStreamEndCapture(side, &body);
    if (le != cudaSuccess) return fail_cuda("launch layer loop body", le);
    if (e != cudaSuccess) return fail_cuda("end layer loop body capture", e);
    if ((e = cudaStreamUpdateCaptureDependencies(st, &node, nullptr, 1,
                                                 cudaStreamSetCaptureDependencies)) != cudaSuccess)
      return fail_cuda("capture dependencies", e);
  }
  for (int l = 0; l < a->n_layers; ++l) {
    if (dev_loop) break;
    if (!per_layer) {
      if (!mark(2 + 3 * l) || !mark(3 + 3 * l) || !mark(4 + 3 * l))
        return fail(SC_ERR_CUDA, "event record", "");
      continue;
    }
    fill_workspace(&p, ws, lay, l & 1);
    p.gathered = nullptr;   // only layer 0 of a host-buffer call counts its rows in
    p.layer = l;
    p.src_base = static_cast<long long>(l) * BLt;
    p.len = a->len + static_cast<size_t>(l) * a->B;
    p.len_out = a->len + static_cast<size_t>(l + 1) * a->B;
    p.pos = a->pos + static_cast<size_t>(l) * BL;
    p.pos_out = a->pos + static_cast<size_t>(l + 1) * BL;
    p.O = a->O != nullptr ? a->O + static_cast<size_t>(l) * BL * a->H * kHeadDim
          : l == a->n_layers - 1 ? o_last : nullptr;
    p.scores = a->scores + static_cast<size_t>(l) * BL;
    p.alpha = a->alpha[l];
    if (l == 0 && (a->pad_mask != nullptr || host_io)) {
      // padding removal may have moved rows: compact layer 0 as well
      gp.src_base = 0;
      gp.layer = 0;
      gp.len = p.len;
      gp.pos = p.pos;
      gp.ident = p.ident;
      gp.gathered = gathered;
      if ((e = launch_gather(gp, st)) != cudaSuccess) return fail_cuda("launch gather kernel", e);
      gp.gathered = nullptr;
      p.gathered = gathered;
      p.gather_target = gather_target;
    }
    if ((e = launch_rows(maps, p, st)) != cudaSuccess) return fail_cuda("launch rows kernel", e);
    if (!mark(2 + 3 * l)) return fail(SC_ERR_CUDA, "event record", "");
    if ((e = launch_cols(maps, p, st)) != cudaSuccess) return fail_cuda("launch cols kernel", e);
    if (!mark(3 + 3 * l)) return fail(SC_ERR_CUDA, "event record", "");
    if (l + 1 < a->n_layers) {
      gp.src_base = static_cast<long long>(l + 1) * BLt;
      gp.layer = l + 1;
      gp.len = p.len_out;
      gp.pos = p.pos_out;
      gp.ident = p.ident_out;
      if ((e = launch_gather(gp, st)) != cudaSuccess) return fail_cuda("launch gather kernel", e);
    }
    if (!mark(4 + 3 * l)) return fail(SC_ERR_CUDA, "event record", "");
  }
  if (use_tail) {
    TailParams tp{};
    tp.n_layers = a->n_layers; tp.B = a->B; tp.L = a->L; tp.H = a->H; tp.w = a->w;
    tp.tail_from = tail_from;
    tp.pos = a->pos;
    tp.len = a->len;
    tp.O = a->O;
    tp.O_last = o_last;
    tp.scores = a->scores;
    tp.status = p.status;
    for (int t = 0; t < 3; ++t) tp.src[t] = src[t];
    tp.src_host = host_io ? 1 : 0;
    if (hres != nullptr) {
      tp.hO = hres->O;
      tp.hO_last = hres->O_last;
      tp.hscores = hres->scores;
      tp.hpos = hres->pos;
      tp.hlen = hres->len;
    }
    tp.n_global = a->n_global;
    for (int g = 0; g < a->n_global; ++g) tp.global_pos[g] = a->global_pos[g];
    for (int l = 0; l < a->n_layers; ++l) tp.alpha[l] = a->alpha[l];
    tp.keep_rule = a->keep_rule;
    if ((e = launch_tail(tp, st)) != cudaSuccess) return fail_cuda("launch tail kernel", e);
  }
  if (!mark(2 + 3 * a->n_layers)) return fail(SC_ERR_CUDA, "event record", "");
  return SC_OK;
}

// ---------------------------------------------------------------------------
// Eager stack calls as CUDA graphs
// ---------------------------------------------------------------------------
// An eager call whose sequences can leave the per-layer kernels for the
// cluster kernel is recorded into a CUDA graph, where the layer loop is a
// device-driven WHILE node (layers that no sequence runs per layer launch
// nothing), and the instantiated graph is launched on the caller's stream.
// Later calls with the same arguments launch the cached graph without
// recording again.  The key holds everything a recorded call reads on the
// host: the sizes, the device addresses, the alpha and global arrays by value,
// the workspace, the device and the process-wide settings read at enqueue
// (rows-kernel design, stall hook).

// Compared and copied as bytes: laid out without padding, zeroed before use.
struct GraphKey {
  unsigned long long stall_ns;
  unsigned long long ws_bytes;
  const void* ptr[16];
  int dev, host_io, flags, n_layers, B, L, H, w, n_global, keep_rule, rows_kernel, unused;
  float alpha[kTailMaxLayers];
  int32_t gpos[SC_MAX_GLOBAL];
};
static_assert(sizeof(GraphKey) == 2 * 8 + 16 * sizeof(void*) + 12 * 4 + kTailMaxLayers * 4 +
                                      SC_MAX_GLOBAL * 4,
              "GraphKey has padding");

struct GraphEntry {
  GraphKey key;
  cudaGraphExec_t exec;
  unsigned long long used;
};

constexpr int kGraphCacheSize = 16;

// Calls recorded into a new graph, and calls that launched a kept one
// (sc_debug_graph_counts).
std::atomic<unsigned long long> g_graphs_recorded{0};
std::atomic<unsigned long long> g_graphs_reused{0};

// A stream of this library per device on which eager calls are recorded
// (nullptr if it cannot be made).
static cudaStream_t record_stream() {
  static std::mutex mu;
  static cudaStream_t rec[256] = {nullptr};
  static bool tried[256] = {false};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 256) {
    cudaGetLastError();
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (!tried[dev]) {
    tried[dev] = true;
    if (cudaStreamCreateWithFlags(&rec[dev], cudaStreamNonBlocking) != cudaSuccess) {
      cudaGetLastError();
      rec[dev] = nullptr;
    }
  }
  return rec[dev];
}

// The key of a stack call (a: the arguments as the kernels see them, with
// device addresses; extra: further addresses the call uses).
static void graph_key(GraphKey* out, const sc_stack_args* a, const void* ws, size_t ws_bytes,
                      bool host_io, const void* const* extra, int n_extra) {
  GraphKey& k = *out;
  std::memset(&k, 0, sizeof(k));
  cudaGetDevice(&k.dev);
  k.host_io = host_io ? 1 : 0;
  k.flags = a->flags;
  k.n_layers = a->n_layers; k.B = a->B; k.L = a->L; k.H = a->H; k.w = a->w;
  k.n_global = a->n_global;
  k.keep_rule = a->keep_rule;
  k.rows_kernel = g_rows_kernel.load(std::memory_order_relaxed);
  k.stall_ns = g_stall_ns.load(std::memory_order_relaxed);
  k.ws_bytes = ws_bytes;
  const void* ptrs[] = {ws, a->Q, a->K, a->V, a->pad_mask, a->O, a->scores, a->pos, a->len,
                        a->O_last};
  int n = 0;
  for (const void* q : ptrs) k.ptr[n++] = q;
  for (int i = 0; i < n_extra && n < 16; ++i) k.ptr[n++] = extra[i];
  for (int l = 0; l < a->n_layers && l < kTailMaxLayers; ++l) k.alpha[l] = a->alpha[l];
  for (int g = 0; g < a->n_global && g < SC_MAX_GLOBAL; ++g) k.gpos[g] = a->global_pos[g];
}

// Launch the graph of `key` on `st`, recording it first (enqueue(stream)
// issues the call's work on a capturing stream) when no cached graph has that
// key.  The least recently used graph makes room for a new one; a graph that
// is still running when it is destroyed is freed when it completes.
static int launch_as_graph(const GraphKey& key, cudaStream_t st,
                           const std::function<int(cudaStream_t)>& enqueue) {
  static std::mutex mu;
  static GraphEntry cache[kGraphCacheSize];
  static int n_cached = 0;
  static unsigned long long clock = 0;
  std::lock_guard<std::mutex> lock(mu);
  ++clock;
  for (int i = 0; i < n_cached; ++i) {
    if (std::memcmp(&cache[i].key, &key, sizeof(key)) == 0) {
      cache[i].used = clock;
      g_graphs_reused.fetch_add(1);
      const cudaError_t e = cudaGraphLaunch(cache[i].exec, st);
      return e == cudaSuccess ? SC_OK : fail_cuda("launch stack graph", e);
    }
  }
  cudaStream_t rec = record_stream();
  if (rec == nullptr) return enqueue(st);   // cannot record: launch the kernels directly
  cudaError_t e = cudaStreamBeginCapture(rec, cudaStreamCaptureModeThreadLocal);
  if (e != cudaSuccess) return fail_cuda("record stack call", e);
  const int rc = enqueue(rec);
  cudaGraph_t g = nullptr;
  e = cudaStreamEndCapture(rec, &g);
  if (rc != SC_OK || e != cudaSuccess) {
    if (g != nullptr) cudaGraphDestroy(g);
    cudaGetLastError();
    return rc != SC_OK ? rc : fail_cuda("end stack call record", e);
  }
  cudaGraphExec_t x = nullptr;
  e = cudaGraphInstantiate(&x, g, 0);
  cudaGraphDestroy(g);
  if (e != cudaSuccess) return fail_cuda("instantiate stack graph", e);
  int slot = n_cached;
  if (n_cached == kGraphCacheSize) {
    slot = 0;
    for (int i = 1; i < n_cached; ++i)
      if (cache[i].used < cache[slot].used) slot = i;
    cudaGraphExecDestroy(cache[slot].exec);
  } else {
    ++n_cached;
  }
  std::memcpy(&cache[slot].key, &key, sizeof(key));
  cache[slot].exec = x;
  cache[slot].used = clock;
  g_graphs_recorded.fetch_add(1);
  e = cudaGraphLaunch(x, st);
  return e == cudaSuccess ? SC_OK : fail_cuda("launch stack graph", e);
}

// Whether a stack call on `st` runs as a graph of this library: eager (the
// stream is not capturing), not asked for plain launches, and with both the
// per-layer kernels and the cluster kernel in its plan.
static bool graph_route(const sc_stack_args* a, cudaStream_t st) {
  if (a->flags & SC_STACK_PLAIN_LAUNCHES) return false;
  bool use_tail = false, per_layer = true;
  if (stack_plan(a, &use_tail, &per_layer) != SC_OK || !(use_tail && per_layer)) return false;
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(st, &cap) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return cap == cudaStreamCaptureStatusNone;
}

int sc_stack_forward(const sc_stack_args* a, void* workspace, size_t ws_bytes, void* stream) {
  if (!a) return SC_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // the checks of stack_forward_impl come first (nothing is recorded for a
  // rejected call): they run again, unchanged, while the call is recorded
  int rc = stack_check(a, workspace, ws_bytes);
  if (rc != SC_OK || !graph_route(a, st))
    return rc != SC_OK ? rc : stack_forward_impl(a, workspace, ws_bytes, stream, nullptr, 0);
  GraphKey key;
  graph_key(&key, a, workspace, ws_bytes, false, nullptr, 0);
  return launch_as_graph(key, st, [&](cudaStream_t s) {
    return stack_forward_impl(a, workspace, ws_bytes, s, nullptr, 0);
  });
}

int sc_stack_forward_profiled(const sc_stack_args* a, void* workspace, size_t ws_bytes,
                              void* stream, void** events, int n_events) {
  if (!a || !events || a->n_layers < 1 || n_events < 3 + 3 * a->n_layers) return SC_ERR_INVALID_ARG;
  return stack_forward_impl(a, workspace, ws_bytes, stream, events, n_events);
}

// ---------------------------------------------------------------------------
// The stack with host inputs and results
// ---------------------------------------------------------------------------

// Device-side copies of a stack's results, after the sc_stack_forward
// workspace: O, scores, pos, len.
struct HostIoLayout {
  size_t O, scores, pos, len, total;
};

static bool host_io_layout(int n_layers, int B, int L, int H, HostIoLayout* h) {
  WsLayout lay;
  if (n_layers < 1 || !ws_layout(B, L, H, &lay)) return false;
  const size_t BL = static_cast<size_t>(B) * L;
  size_t off = align_up(lay.total);
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align_up(off + bytes);
    return at;
  };
  h->O = take(sizeof(uint16_t) * n_layers * BL * H * kHeadDim);
  h->scores = take(sizeof(float) * n_layers * BL);
  h->pos = take(sizeof(int32_t) * (n_layers + 1) * BL);
  h->len = take(sizeof(int32_t) * (n_layers + 1) * B);
  h->total = off;
  return true;
}

// The device address of page-locked host memory [p, p + bytes), or nullptr
// unless both ends of the range are page-locked host memory mapped for the
// device at consecutive addresses (so a kernel may read or write all of it).
static void* mapped_host_range(const void* p, size_t bytes) {
  if (p == nullptr || bytes == 0) return nullptr;
  const char* first = static_cast<const char*>(p);
  const char* last = first + (bytes - 1);
  cudaPointerAttributes a0{}, a1{};
  if (cudaPointerGetAttributes(&a0, first) != cudaSuccess ||
      cudaPointerGetAttributes(&a1, last) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  if (a0.type != cudaMemoryTypeHost || a1.type != cudaMemoryTypeHost ||
      a0.devicePointer == nullptr || a1.devicePointer == nullptr)
    return nullptr;
  char* d0 = static_cast<char*>(a0.devicePointer);
  if (static_cast<char*>(a1.devicePointer) != d0 + (bytes - 1)) return nullptr;
  return d0;
}

size_t sc_stack_host_workspace_size(int n_layers, int B, int L, int H) {
  HostIoLayout h;
  if (!host_io_layout(n_layers, B, L, H, &h)) return 0;
  return h.total;
}

int sc_stack_forward_host(const sc_stack_args* a, void* workspace, size_t ws_bytes, void* stream) {
  if (!a) return SC_ERR_INVALID_ARG;
  if (a->n_layers < 1 || (a->flags & ~(SC_STACK_NO_TAIL | SC_STACK_PLAIN_LAUNCHES)))
    return SC_ERR_INVALID_ARG;
  int rc = check_common(a->B, a->L, a->H, a->w, a->global_pos, a->n_global);
  if (rc != SC_OK) return rc;
  if (!a->Q || !a->K || !a->V || !a->alpha || !a->scores || !a->pos || !a->len)
    return SC_ERR_INVALID_ARG;
  HostIoLayout hl;
  if (!host_io_layout(a->n_layers, a->B, a->L, a->H, &hl)) return SC_ERR_INVALID_ARG;
  if (!workspace || ws_bytes < hl.total || (reinterpret_cast<uintptr_t>(workspace) % kAlign))
    return SC_ERR_WORKSPACE;
  const size_t BL = static_cast<size_t>(a->B) * a->L;
  const size_t qkv_bytes = sizeof(uint16_t) * a->n_layers * BL * a->H * kHeadDim;
  void* q = mapped_host_range(a->Q, qkv_bytes);
  void* k = mapped_host_range(a->K, qkv_bytes);
  void* v = mapped_host_range(a->V, qkv_bytes);
  // O of every layer, or (O == NULL) only the last layer's to O_last, or none
  const size_t layer_o_bytes = qkv_bytes / a->n_layers;
  void* o = a->O ? mapped_host_range(a->O, qkv_bytes) : nullptr;
  void* o_last = !a->O && a->O_last ? mapped_host_range(a->O_last, layer_o_bytes) : nullptr;
  void* sc = mapped_host_range(a->scores, sizeof(float) * a->n_layers * BL);
  void* ps = mapped_host_range(a->pos, sizeof(int32_t) * (a->n_layers + 1) * BL);
  void* ln = mapped_host_range(a->len, sizeof(int32_t) * (a->n_layers + 1) * a->B);
  void* pm = a->pad_mask ? mapped_host_range(a->pad_mask, BL) : nullptr;
  if (!q || !k || !v || (a->O && !o) || (!a->O && a->O_last && !o_last) || !sc || !ps || !ln ||
      (a->pad_mask && !pm))
    return fail(SC_ERR_INVALID_ARG, "sc_stack_forward_host",
                "a host buffer is not page-locked memory mapped for the device");
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(o) || !aligned16(o_last) ||
      (reinterpret_cast<uintptr_t>(sc) & 3u) || (reinterpret_cast<uintptr_t>(ps) & 3u) ||
      (reinterpret_cast<uintptr_t>(ln) & 3u))
    return SC_ERR_INVALID_ARG;
  char* ws = static_cast<char*>(workspace);
  sc_stack_args d = *a;
  d.Q = static_cast<const uint16_t*>(q);
  d.K = static_cast<const uint16_t*>(k);
  d.V = static_cast<const uint16_t*>(v);
  d.pad_mask = static_cast<const uint8_t*>(pm);
  uint16_t* const dO = reinterpret_cast<uint16_t*>(ws + hl.O);
  d.O = a->O ? dO : nullptr;
  d.O_last = a->O ? nullptr
             : a->O_last ? dO + (a->n_layers - 1) * (layer_o_bytes / sizeof(uint16_t)) : nullptr;
  d.scores = reinterpret_cast<float*>(ws + hl.scores);
  d.pos = reinterpret_cast<int32_t*>(ws + hl.pos);
  d.len = reinterpret_cast<int32_t*>(ws + hl.len);
  const HostResults hres{static_cast<uint16_t*>(o), static_cast<uint16_t*>(o_last),
                         static_cast<float*>(sc), static_cast<int32_t*>(ps),
                         static_cast<int32_t*>(ln)};
  // the stack, then the export of the per-layer results, on stream s
  auto enqueue = [&](cudaStream_t s) -> int {
    int rc2 = stack_forward_impl(&d, workspace, hl.O, s, nullptr, 0, true, &hres);
    if (rc2 != SC_OK) return rc2;
    bool use_tail = false, per_layer = true;
    if ((rc2 = stack_plan(a, &use_tail, &per_layer)) != SC_OK) return rc2;
    int dev = 0, sms = 0;
    cudaError_t ce = cudaGetDevice(&dev);
    if (ce == cudaSuccess) ce = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (ce != cudaSuccess) return fail_cuda("device attributes", ce);
    WsLayout lay;
    ws_layout(a->B, a->L, a->H, &lay);
    ExportParams e{};
    e.n_layers = a->n_layers; e.B = a->B; e.L = a->L; e.H = a->H;
    e.O = dO; e.scores = d.scores; e.pos = d.pos; e.len = d.len;
    e.hO = static_cast<uint16_t*>(o);
    e.hO_last = static_cast<uint16_t*>(o_last);
    e.hscores = static_cast<float*>(sc);
    e.hpos = static_cast<int32_t*>(ps);
    e.hlen = static_cast<int32_t*>(ln);
    e.tail_from = reinterpret_cast<const int32_t*>(ws + lay.tail_from);
    if (use_tail) {
      // the per-layer results go out beside the cluster kernel, on the SMs it
      // leaves idle (one CTA per SM fits beside one of its CTAs); the cluster
      // kernel writes its own layers' results to the host buffers itself.  The
      // export ends with a grid wait, so the call ends after the cluster kernel.
      e.part = 1;
      if ((ce = launch_export(e, sms, s)) != cudaSuccess)
        return fail_cuda("launch export kernel", ce);
    } else {
      e.part = 0;
      if ((ce = launch_export(e, 4 * sms, s)) != cudaSuccess)
        return fail_cuda("launch export kernel", ce);
    }
    return SC_OK;
  };
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if ((rc = stack_check(&d, workspace, hl.O)) != SC_OK) return rc;
  if (!graph_route(a, st)) return enqueue(st);
  const void* results[] = {o, o_last, sc, ps, ln};
  GraphKey key;
  graph_key(&key, &d, workspace, ws_bytes, true, results, 5);
  return launch_as_graph(key, st, enqueue);
}

int sc_stack_host_launch_count(const sc_stack_args* a, int* count) {
  if (!a || !count) return SC_ERR_INVALID_ARG;
  if (a->n_layers < 1 || (a->flags & ~(SC_STACK_NO_TAIL | SC_STACK_PLAIN_LAUNCHES)))
    return SC_ERR_INVALID_ARG;
  int rc = check_common(a->B, a->L, a->H, a->w, a->global_pos, a->n_global);
  if (rc != SC_OK) return rc;
  if ((rc = ensure_configured()) != SC_OK) return rc;
  bool use_tail = false, per_layer = true;
  if ((rc = stack_plan(a, &use_tail, &per_layer)) != SC_OK) return rc;
  int k = 2;   // padding removal / global lookup, and the export
  if (per_layer) k += 1 + 2 * a->n_layers + (a->n_layers - 1);
  if (use_tail) k += 1;   // the cluster kernel (it writes its own layers' results)
  *count = k;
  return SC_OK;
}

int sc_stack_launch_count(const sc_stack_args* a, int* count) {
  if (!a || !count) return SC_ERR_INVALID_ARG;
  if (a->n_layers < 1 || (a->flags & ~(SC_STACK_NO_TAIL | SC_STACK_PLAIN_LAUNCHES)))
    return SC_ERR_INVALID_ARG;
  int rc = check_common(a->B, a->L, a->H, a->w, a->global_pos, a->n_global);
  if (rc != SC_OK) return rc;
  if ((rc = ensure_configured()) != SC_OK) return rc;
  bool use_tail = false, per_layer = true;
  if ((rc = stack_plan(a, &use_tail, &per_layer)) != SC_OK) return rc;
  int k = 1;   // padding removal / global lookup
  if (per_layer) k += (a->pad_mask ? 1 : 0) + 2 * a->n_layers + (a->n_layers - 1);
  if (use_tail) k += 1;
  *count = k;
  return SC_OK;
}

void sc_debug_stall_waits(unsigned long long ns) { g_stall_ns.store(ns); }

void sc_debug_graph_counts(unsigned long long* recorded, unsigned long long* reused) {
  if (recorded) *recorded = g_graphs_recorded.load();
  if (reused) *reused = g_graphs_reused.load();
}

int sc_select_rows_kernel(int which) {
  if (which != SC_ROWS_SINGLE_PASS && which != SC_ROWS_TWO_PASS) return SC_ERR_INVALID_ARG;
  g_rows_kernel.store(which);
  return SC_OK;
}

int sc_workspace_status(void* workspace, size_t ws_bytes, void* stream) {
  if (!workspace || ws_bytes < kAlign) return SC_ERR_WORKSPACE;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(st) != cudaSuccess) return SC_ERR_CUDA;
  int word = 0;
  if (cudaMemcpy(&word, workspace, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
    return SC_ERR_CUDA;
  if (word == 0) return SC_OK;
  if (cudaMemset(workspace, 0, sizeof(int)) != cudaSuccess) return SC_ERR_CUDA;
  return (word & kStatusTimeout) ? SC_ERR_TIMEOUT : SC_ERR_CUDA;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Single layer without any allocation by the caller or the library.
// ---------------------------------------------------------------------------
// Some callers cannot allocate device memory where they run a layer: hosts
// whose whole device heap belongs to another allocator that exposes no hook
// (plugins inside other frameworks), deployments with a fixed memory budget
// that forbid allocation after start-up, and latency-critical services that
// cannot afford cudaMalloc's implicit device synchronisation.  For them the
// scratch of one layer lives in this fixed array, held by every GPU that loads
// the library until the process exits.
namespace {

constexpr size_t kStaticWorkspaceBytes = size_t(6) << 20;  // 6 MiB

}  // namespace

static __device__ __align__(256) unsigned char g_static_workspace[kStaticWorkspaceBytes];

namespace {

// Device address of g_static_workspace on the current device.  In host code
// the array's name is only a stand-in, so the address is looked up once per
// device (with that device current) and cached.
int static_workspace(char** out) {
  static std::mutex mu;
  static void* addr[256] = {nullptr};
  int dev = 0;
  const cudaError_t ge = cudaGetDevice(&dev);
  if (ge != cudaSuccess) return fail_cuda("cudaGetDevice", ge);
  if (dev < 0 || dev >= 256) return fail(SC_ERR_CUDA, "cudaGetDevice", "device index out of range");
  std::lock_guard<std::mutex> lock(mu);
  if (addr[dev] == nullptr) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_static_workspace);
    if (e != cudaSuccess) return fail_cuda("static workspace address", e);
    addr[dev] = p;
  }
  *out = static_cast<char*>(addr[dev]);
  return SC_OK;
}

}  // namespace

extern "C" int sc_layer_forward_noalloc(const sc_layer_args* a, void* stream) {
  if (!a) return SC_ERR_INVALID_ARG;
  int rc = check_common(a->B, a->L, a->H, a->w, a->global_pos, a->n_global);
  if (rc != SC_OK) return rc;
  if (!a->Q || !a->K || !a->V || !a->len || !a->pos || !a->O || !a->scores || !a->pos_out ||
      !a->len_out)
    return SC_ERR_INVALID_ARG;
  if (!aligned16(a->Q) || !aligned16(a->K) || !aligned16(a->V) || !aligned16(a->O))
    return SC_ERR_INVALID_ARG;
  if (a->pos_out == a->pos || a->len_out == a->len) return SC_ERR_INVALID_ARG;
  if ((rc = check_keep(a->keep_rule, &a->alpha, 1, a->theta)) != SC_OK) return rc;
  // a single layer reads its rows in place, so the compacted copies that the
  // layout reserves last are not needed: everything before them must fit
  WsLayout lay;
  ws_layout(a->B, a->L, a->H, &lay);
  if (lay.qkv > kStaticWorkspaceBytes) {
    char d[128];
    snprintf(d, sizeof d, "B=%d, L=%d, H=%d need %zu bytes of scratch, the static array holds %zu",
             a->B, a->L, a->H, lay.qkv, kStaticWorkspaceBytes);
    return fail(SC_ERR_UNSUPPORTED, "sc_layer_forward_noalloc", d);
  }
  if ((rc = ensure_configured()) != SC_OK) return rc;
  char* ws = nullptr;
  if ((rc = static_workspace(&ws)) != SC_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);

  // the compacted-row descriptors point at the caller's tensors: never read here
  TensorMaps maps;
  const uint16_t* src[3] = {a->Q, a->K, a->V};
  uint16_t* const cmp[3] = {const_cast<uint16_t*>(a->Q), const_cast<uint16_t*>(a->K),
                            const_cast<uint16_t*>(a->V)};
  const long long tokens = static_cast<long long>(a->B) * a->L;
  if (!encode_maps(&maps, src, tokens, cmp, tokens, a->H)) return SC_ERR_CUDA;
  // the array keeps the previous call's contents: clear the counters, which
  // must start at zero (the status word is kept until sc_layer_noalloc_status
  // reads it, so that an expired wait of any call is reported)
  cudaError_t e;
  if ((rc = reset_counters(ws, lay, st)) != SC_OK) return rc;

  LayerParams p{};
  p.B = a->B; p.L = a->L; p.H = a->H; p.w = a->w;
  p.T = (a->L + kTile - 1) / kTile;
  p.src_base = 0;
  p.len = a->len;
  p.pos = a->pos;
  p.O = a->O;
  p.scores = a->scores;
  p.pos_out = a->pos_out;
  p.len_out = a->len_out;
  p.alpha = a->alpha;
  p.theta = a->theta;
  p.keep_rule = a->keep_rule;
  fill_workspace(&p, ws, lay, 0);

  PrepParams pp{};
  pp.B = a->B; pp.L = a->L;
  pp.pos_in = a->pos;
  pp.len_in = a->len;
  pp.gcur = const_cast<int32_t*>(p.gcur);
  pp.ng = const_cast<int32_t*>(p.ng);
  pp.ident = const_cast<int32_t*>(p.ident);
  pp.n_global = a->n_global;
  for (int g = 0; g < a->n_global; ++g) pp.global_pos[g] = a->global_pos[g];
  if ((e = launch_prep(pp, st)) != cudaSuccess) return fail_cuda("launch prep kernel", e);
  if ((e = launch_rows(maps, p, st)) != cudaSuccess) return fail_cuda("launch rows kernel", e);
  if ((e = launch_cols(maps, p, st)) != cudaSuccess) return fail_cuda("launch cols kernel", e);
  return SC_OK;
}

extern "C" int sc_layer_noalloc_status(void* stream) {
  char* ws = nullptr;
  int rc = static_workspace(&ws);
  if (rc != SC_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaStreamSynchronize(st) != cudaSuccess) return SC_ERR_CUDA;
  int word = 0;
  if (cudaMemcpy(&word, ws, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
    return SC_ERR_CUDA;
  if (word == 0) return SC_OK;
  if (cudaMemset(ws, 0, sizeof(int)) != cudaSuccess) return SC_ERR_CUDA;
  return (word & kStatusTimeout) ? SC_ERR_TIMEOUT : SC_ERR_CUDA;
}

// ---------------------------------------------------------------------------
// the encoder layer around the path: GEMMs, layer norms, the layer driver
// ---------------------------------------------------------------------------
namespace {

bool aligned_ptr16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Fills the GEMM parameters and descriptors for out = act(A[a_idx] W^T + b) (+ res[res_idx]).
int make_gemm(GemmParams* g, int B, int L, int N, int K, const uint16_t* A, const int32_t* rows,
              const int32_t* a_idx, const uint16_t* W, const float* bias, int gelu,
              const uint16_t* res, const int32_t* res_idx, void* out, int out_f32, int* status) {
  *g = GemmParams{};
  // Column-tile width: with a gathered A, 256 (A is fetched again for every
  // column tile); otherwise the width among 256, 192 and 128 (dividing N) with
  // the least (whole rounds of tiles over the SMs) x (width + 32), the 32 a
  // per-tile cost in columns' worth of time.  The row count is a bound (rows
  // are counted on the device).
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
    cudaGetLastError();
    sms = 152;
  }
  const long long row_tiles = static_cast<long long>(B) * ((L + kTile - 1) / kTile);
  int bn = 256;
  if (!a_idx) {
    long long best = -1;
    for (int c : {256, 192, 128}) {
      if (c != 256 && N % c != 0) continue;
      const long long tiles = row_tiles * ((N + c - 1) / c);
      const long long cost = (tiles + sms - 1) / sms * (c + 32);
      if (best < 0 || cost < best) {
        best = cost;
        bn = c;
      }
    }
  }
  const int wbox = N < bn ? N : bn;
  if (!encode_2d(&g->map_a, A, static_cast<long long>(B) * L, K, 1) ||
      !encode_2d(&g->map_at, A, static_cast<long long>(B) * L, K, kTile) ||
      !encode_2d(&g->map_w, W, N, K, wbox))
    return SC_ERR_CUDA;
  g->B = B; g->L = L; g->N = N; g->K = K; g->bn = bn; g->wbox = wbox;
  g->rows = rows; g->a_idx = a_idx; g->bias = bias; g->gelu = gelu;
  g->res = res; g->res_idx = res_idx;
  g->out = out; g->out_f32 = out_f32; g->out_split = 0;
  g->status = status;
  return SC_OK;
}

struct EncLayout {
  size_t attn, qkv, kept, s, h1, f, total;
};

bool enc_layout(int B, int L, int H, EncLayout* e) {
  WsLayout lay;
  if (!ws_layout(B, L, H, &lay)) return false;
  const size_t rows = static_cast<size_t>(B) * L, D = static_cast<size_t>(H) * kHeadDim;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off = align_up(off + bytes);
    return at;
  };
  e->attn = take(lay.total);
  e->qkv = take(3 * rows * D * sizeof(uint16_t));
  e->kept = take(rows * sizeof(int32_t));
  e->s = take(rows * D * sizeof(float));
  e->h1 = take(rows * D * sizeof(uint16_t));
  e->f = take(rows * 4 * D * sizeof(uint16_t));
  e->total = off;
  return true;
}

}  // namespace

extern "C" size_t sc_encoder_workspace_size(int B, int L, int H) {
  if (B < 1 || L < 1 || H < 2 || (H & 1) || H > kTailMaxHeads || L > kMaxLen) return 0;
  EncLayout e;
  return enc_layout(B, L, H, &e) ? e.total : 0;
}

extern "C" int sc_linear_forward(const sc_linear_args* a, void* workspace, size_t ws_bytes,
                                 void* stream) {
  if (!a) return SC_ERR_INVALID_ARG;
  if (a->B < 1 || a->L < 1 || a->N < kTile || a->N % kTile || a->K < 64 || a->K % 64 ||
      a->K > 8192 || static_cast<long long>(a->B) * a->L > (1ll << 31) - 1)
    return SC_ERR_INVALID_ARG;
  if (!a->A || !a->W || !a->out || !aligned_ptr16(a->A) || !aligned_ptr16(a->W) ||
      !aligned_ptr16(a->out) || (a->res && !aligned_ptr16(a->res)))
    return SC_ERR_INVALID_ARG;
  if (!workspace || ws_bytes < kAlign || (reinterpret_cast<uintptr_t>(workspace) % kAlign))
    return SC_ERR_WORKSPACE;
  int rc = ensure_configured();
  if (rc != SC_OK) return rc;
  GemmParams g;
  if ((rc = make_gemm(&g, a->B, a->L, a->N, a->K, a->A, a->rows, a->gidx, a->W, a->bias, a->gelu,
                      a->res, a->res_gathered ? a->gidx : nullptr, a->out, a->out_f32,
                      static_cast<int*>(workspace))) != SC_OK)
    return rc;
  const cudaError_t e = launch_gemm(g, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? SC_OK : fail_cuda("launch gemm kernel", e);
}

extern "C" int sc_layer_norm_forward(int B, int L, int D, const int32_t* rows, const float* in,
                                     const float* gamma, const float* beta, float eps,
                                     uint16_t* out, void* stream) {
  if (B < 1 || L < 1 || D < 32 || D % 32 || D > 1024 || !in || !gamma || !beta || !out ||
      !(eps > 0.f))
    return SC_ERR_INVALID_ARG;
  int rc = ensure_configured();
  if (rc != SC_OK) return rc;
  LayerNormParams q{B, L, D, rows, in, gamma, beta, eps, out};
  const cudaError_t e = launch_layernorm(q, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? SC_OK : fail_cuda("launch layer-norm kernel", e);
}

extern "C" int sc_encoder_layer_forward(const sc_encoder_args* a, void* workspace, size_t ws_bytes,
                                        void* stream) {
  if (!a) return SC_ERR_INVALID_ARG;
  if (a->H < 2 || (a->H & 1) || a->H > kTailMaxHeads) return SC_ERR_UNSUPPORTED;
  int rc = check_common(a->B, a->L, a->H, a->w, a->global_pos, a->n_global);
  if (rc != SC_OK) return rc;
  if ((rc = check_keep(a->keep_rule, &a->alpha, 1, a->theta)) != SC_OK) return rc;
  const void* need[] = {a->X, a->len, a->pos, a->W_qkv, a->b_qkv, a->W_o, a->b_o, a->ln1_gamma,
                        a->ln1_beta, a->W_1, a->b_1, a->W_2, a->b_2, a->ln2_gamma, a->ln2_beta,
                        a->Y, a->O, a->scores, a->pos_out, a->len_out};
  for (const void* q : need)
    if (!q) return SC_ERR_INVALID_ARG;
  const void* al[] = {a->X, a->W_qkv, a->W_o, a->W_1, a->W_2, a->Y, a->O};
  for (const void* q : al)
    if (!aligned_ptr16(q)) return SC_ERR_INVALID_ARG;
  if (a->pos_out == a->pos || a->len_out == a->len) return SC_ERR_INVALID_ARG;
  EncLayout el;
  if (!enc_layout(a->B, a->L, a->H, &el)) return SC_ERR_UNSUPPORTED;
  if (!workspace || ws_bytes < el.total || (reinterpret_cast<uintptr_t>(workspace) % kAlign))
    return SC_ERR_WORKSPACE;
  if ((rc = ensure_configured()) != SC_OK) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  char* ws = static_cast<char*>(workspace);
  const int B = a->B, L = a->L, D = a->H * kHeadDim;
  const size_t rows = static_cast<size_t>(B) * L;
  uint16_t* qkv = reinterpret_cast<uint16_t*>(ws + el.qkv);
  uint16_t* Qb = qkv;
  uint16_t* Kb = qkv + rows * D;
  uint16_t* Vb = qkv + 2 * rows * D;
  int32_t* kept = reinterpret_cast<int32_t*>(ws + el.kept);
  float* S = reinterpret_cast<float*>(ws + el.s);
  uint16_t* H1 = reinterpret_cast<uint16_t*>(ws + el.h1);
  uint16_t* F = reinterpret_cast<uint16_t*>(ws + el.f);
  int* status = reinterpret_cast<int*>(ws + el.attn);   // the attention workspace's status word
  cudaError_t e;

  // Q, K, V of the current tokens: one GEMM, its column blocks split by tensor
  GemmParams g;
  if ((rc = make_gemm(&g, B, L, 3 * D, D, a->X, a->len, nullptr, a->W_qkv, a->b_qkv, 0, nullptr,
                      nullptr, nullptr, 0, status)) != SC_OK)
    return rc;
  g.out_split = D;
  g.outs[0] = Qb; g.outs[1] = Kb; g.outs[2] = Vb;
  if ((e = launch_gemm(g, st)) != cudaSuccess) return fail_cuda("launch QKV gemm", e);

  // sparse attention with token pruning; the kept tokens' current indices
  sc_layer_args la{};
  la.B = B; la.L = L; la.H = a->H; la.w = a->w;
  la.Q = Qb; la.K = Kb; la.V = Vb;
  la.len = a->len; la.pos = a->pos;
  la.global_pos = a->global_pos; la.n_global = a->n_global;
  la.alpha = a->alpha; la.theta = a->theta; la.keep_rule = a->keep_rule;
  la.O = a->O; la.scores = a->scores; la.pos_out = a->pos_out; la.len_out = a->len_out;
  WsLayout lay;
  ws_layout(B, L, a->H, &lay);
  if ((rc = layer_forward_impl(&la, ws + el.attn, lay.total, stream, kept)) != SC_OK) return rc;

  // S1 = X[kept] + O[kept] W_o^T + b_o: the kept rows of O are compacted once
  // (into F's space, unused until the feed-forward block) so that the GEMM reads
  // A with tiled copies; X[kept] is gathered row by row in its epilogue
  RowGatherParams rg{B, L, D, a->len_out, kept, a->O, F};
  if ((e = launch_row_gather(rg, st)) != cudaSuccess) return fail_cuda("launch row gather", e);
  if ((rc = make_gemm(&g, B, L, D, D, F, a->len_out, nullptr, a->W_o, a->b_o, 0, a->X, kept, S, 1,
                      status)) != SC_OK)
    return rc;
  if ((e = launch_gemm(g, st)) != cudaSuccess) return fail_cuda("launch output gemm", e);
  LayerNormParams ln{B, L, D, a->len_out, S, a->ln1_gamma, a->ln1_beta, 1e-5f, H1};
  if ((e = launch_layernorm(ln, st)) != cudaSuccess) return fail_cuda("launch layer norm 1", e);
  // the feed-forward block on the kept tokens
  if ((rc = make_gemm(&g, B, L, 4 * D, D, H1, a->len_out, nullptr, a->W_1, a->b_1, 1, nullptr,
                      nullptr, F, 0, status)) != SC_OK)
    return rc;
  if ((e = launch_gemm(g, st)) != cudaSuccess) return fail_cuda("launch ffn gemm 1", e);
  if ((rc = make_gemm(&g, B, L, D, 4 * D, F, a->len_out, nullptr, a->W_2, a->b_2, 0, H1, nullptr,
                      S, 1, status)) != SC_OK)
    return rc;
  if ((e = launch_gemm(g, st)) != cudaSuccess) return fail_cuda("launch ffn gemm 2", e);
  ln.gamma = a->ln2_gamma; ln.beta = a->ln2_beta; ln.out = a->Y;
  if ((e = launch_layernorm(ln, st)) != cudaSuccess) return fail_cuda("launch layer norm 2", e);
  return SC_OK;
}
