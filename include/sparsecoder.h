/*
 * sparsecoder.h -- C ABI of the GB300 (sm_103a) hot path of SparseCoder
 * (arXiv 2310.07109): Longformer-style sparse attention fused with learned
 * token pruning, one layer or a pruned stack of layers.
 *
 * Conventions
 * -----------
 * - All tensors are caller-owned DEVICE memory unless a field says "host".
 *   The library allocates nothing; scratch lives in a caller-supplied
 *   workspace of sc_workspace_size() bytes (device memory, 256-byte aligned).
 * - bf16 tensors are passed as uint16_t bit patterns.  Q/K/V/O rows are
 *   [.., token, head, 64] with the head dimension fixed at SC_HEAD_DIM = 64;
 *   every such pointer must be 16-byte aligned.
 * - Every call is asynchronous on `stream` (a cudaStream_t passed as void*;
 *   NULL = legacy default stream).  No call synchronises the host, and no
 *   current length ever travels back to the host: layer l+1 reads the
 *   lengths layer l wrote, on the device.
 * - Arguments are validated on the host before anything is launched; a bad
 *   argument returns an SC_ERR_* code with nothing enqueued.  CUDA launch
 *   errors return SC_ERR_CUDA.  No C++ exception crosses this interface.
 * - Every wait inside a kernel is bounded (about 2 s).  A wait that expires
 *   makes the kernel record SC_ERR_TIMEOUT in the workspace status word and
 *   return; sc_workspace_status() reports (and clears) it.
 *
 * The method (paper sections / equations cited on each call):
 *   current tokens c = 0..n-1 of one sequence, original positions p(c);
 *   G = global original positions; a token is global when p(c) is in G.
 *   Allowed keys of row i: all n tokens if i is global, otherwise
 *   {j : |i - j| <= w} U {global j}  (Sec. "Sparse Attention": unit i is
 *   attended by units i-w..i+w; Sec. "Extractor of Attention Scores": special
 *   tokens attend to every token and are attended by every token).
 *   P_h = row-wise softmax of q.k / sqrt(64) over the allowed keys (Fig. 1
 *   caption); O_h[i] = sum_j P_h[i,j] v_j.
 *   s_j = (1/(H n)) sum_h sum_i P_h[i,j]: probabilities accumulated
 *   vertically (Sec. "Pruning"; Fig. 1 caption), averaged over heads and rows.
 *   keep_j = (j == 0) || s_j >= theta  (Sec. "Token Pruning", Step 2, the
 *   binarised mask, read as >= and with the first token always kept);
 *   kept tokens are compacted in order (Step 3, hard pruning).
 *   Keep rules (sc_keep_rule): theta = alpha / n per sequence (default),
 *   an absolute theta (the schedule of Sec. "RQ4": thresholds scaled linearly
 *   with depth), or the "top-k of the sequence length" family of Sec.
 *   "Pruning": a layer keeps k = ceil(rho n) tokens, clamped to 1..n, the
 *   first token and the k-1 others with the largest s_j, ties to the lower
 *   current index.
 */
#ifndef SPARSECODER_H
#define SPARSECODER_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define SC_HEAD_DIM 64
#define SC_MAX_LEN 4096   /* longest supported (padded) sequence */
#define SC_MAX_GLOBAL 16  /* most global positions per call */
#define SC_MAX_WINDOW 512 /* widest one-sided window when L > 640 */
#define SC_TAIL_MAX_LEN 384 /* sequences this short finish in the cluster kernel (see sc_stack_forward) */

typedef enum {
  SC_OK = 0,
  SC_ERR_INVALID_ARG = 1, /* null pointer, bad size, misaligned pointer, bad global set */
  SC_ERR_UNSUPPORTED = 2, /* L > SC_MAX_LEN, too many globals, window too wide */
  SC_ERR_CUDA = 3,        /* a CUDA runtime/driver call failed */
  SC_ERR_TIMEOUT = 4,     /* a bounded device-side wait expired (from sc_workspace_status) */
  SC_ERR_WORKSPACE = 5    /* workspace missing, too small or misaligned */
} sc_status;

/* What decides that a token survives a layer (the value `alpha` of a layer). */
typedef enum {
  SC_KEEP_RELATIVE = 0,  /* s_j >= alpha / n (theta = alpha / n per sequence) */
  SC_KEEP_ABSOLUTE = 1,  /* s_j >= alpha (an absolute threshold) */
  SC_KEEP_TOP_RATIO = 2  /* the ceil(alpha n) best tokens (alpha = kept ratio; k is
                            computed in double from the float alpha, so exactly) */
} sc_keep_rule;

/*
 * One layer on tokens already in current (compacted) order.
 *
 * Q, K, V    bf16 [B][L][H][64]; row c of sequence b holds current token c.
 *            Rows at or beyond len[b] are never read.
 * len        int32 [B]: current length n_b (0 <= n_b <= L).
 * pos        int32 [B][L]: original position of each current token, strictly
 *            increasing within [0, n_b).  Decides which tokens are global and
 *            is what pos_out is compacted from.
 * w          one-sided window (>= 0).
 * global_pos HOST int32 [n_global]: sorted, distinct original positions,
 *            0 <= g < L, n_global <= SC_MAX_GLOBAL (may be 0).
 * alpha      the keep rule's value: theta_b = alpha / n_b (SC_KEEP_RELATIVE;
 *            the threshold schedule of Sec. "RQ4" scales it linearly across
 *            layers, the caller supplies this layer's), theta_b = alpha
 *            (SC_KEEP_ABSOLUTE), or the kept ratio (SC_KEEP_TOP_RATIO; finite).
 *            Ignored when theta != NULL.
 * theta      optional float [B]: absolute thresholds per sequence (threshold
 *            rules only; must be NULL under SC_KEEP_TOP_RATIO).
 * O          bf16 [B][L][H][64] out: attention output of every current token
 *            (all n_b tokens, before pruning) at its current slot.
 * scores     float [B][L] out: s_j at current slot j.
 * pos_out    int32 [B][L] out: original positions of the kept tokens, in order.
 * len_out    int32 [B] out: number of kept tokens.
 * keep_rule  an sc_keep_rule (0 = SC_KEEP_RELATIVE).
 * Slots at or beyond the current (resp. kept) length are left untouched.
 * pos_out/len_out must not alias pos/len.
 */
typedef struct {
  int B, L, H, w;
  const uint16_t* Q;
  const uint16_t* K;
  const uint16_t* V;
  const int32_t* len;
  const int32_t* pos;
  const int32_t* global_pos;
  int n_global;
  float alpha;
  const float* theta;
  uint16_t* O;
  float* scores;
  int32_t* pos_out;
  int32_t* len_out;
  int keep_rule;
} sc_layer_args;

/*
 * A pruned stack of n_layers layers over inputs in ORIGINAL-position order.
 *
 * Q, K, V    bf16 [n_layers][B][L][H][64]: layer l reads, for each token that
 *            survived layers 0..l-1, the row at its original position.
 * pad_mask   uint8 [B][L] (1 = real token) or NULL (no padding).  Padding
 *            tokens are removed before layer 0 (Fig. "experiment" caption:
 *            shorter inputs are padded to max_length).
 * w, global_pos, n_global   as for sc_layer_args.
 * alpha      HOST float [n_layers]: the keep rule's value per layer:
 *            theta_{l,b} = alpha[l] / n_{l,b} (SC_KEEP_RELATIVE), theta_l =
 *            alpha[l] (SC_KEEP_ABSOLUTE) or the kept ratio rho_l
 *            (SC_KEEP_TOP_RATIO; finite).
 * O          bf16 [n_layers][B][L][H][64] out (current slots of each layer), or
 *            NULL: then no layer's O is written but the last layer's, to O_last.
 * scores     float [n_layers][B][L] out.
 * pos        int32 [n_layers+1][B][L] out: pos[0] = real tokens after padding
 *            removal, pos[l+1] = survivors of layer l.
 * len        int32 [n_layers+1][B] out.
 * flags      0, or a combination of SC_STACK_NO_TAIL: run every layer of every
 *            sequence through the per-layer kernels, and SC_STACK_PLAIN_LAUNCHES:
 *            launch the kernels directly on the stream even when the call is
 *            not being captured (see sc_stack_forward).
 * keep_rule  an sc_keep_rule (0 = SC_KEEP_RELATIVE), the same for every layer.
 * O_last     used only when O is NULL: bf16 [B][L][H][64] out, the last layer's
 *            O at its current slots; or NULL as well (no O is written at all,
 *            which saves the 1536 bytes per token and layer of O stores).
 *            Earlier layers' O is not needed to decide the kept tokens, whose
 *            scores come from the probabilities alone (Sec. "Token Pruning").
 */
#define SC_STACK_NO_TAIL 1
#define SC_STACK_PLAIN_LAUNCHES 2

typedef struct {
  int n_layers, B, L, H, w;
  const uint16_t* Q;
  const uint16_t* K;
  const uint16_t* V;
  const uint8_t* pad_mask;
  const int32_t* global_pos;
  int n_global;
  const float* alpha;
  uint16_t* O;
  float* scores;
  int32_t* pos;
  int32_t* len;
  int flags;
  int keep_rule;
  uint16_t* O_last;
} sc_stack_args;

/*
 * sc_layer_forward without any device allocation, by the caller or the
 * library: for callers that cannot allocate device memory where they run a
 * layer -- hosts whose device heap belongs to another allocator without a hook
 * for plugins, deployments with a fixed memory budget that forbid allocation
 * after start-up, and latency-critical services that cannot afford the
 * implicit device synchronisation of cudaMalloc.  The paper has no
 * counterpart; this is an interface convenience.
 *
 * Same arguments, semantics and results as sc_layer_forward (the caller still
 * passes every input and output).  The scratch comes from a 6 MiB array
 * compiled into the library, which every GPU that loads it holds until the
 * process exits; sizes whose scratch does not fit (from roughly B*L*H = 100k
 * (sequence, token, head) rows on; B=2, L=4096, H=12 is 98k and fits) return
 * SC_ERR_UNSUPPORTED with the detail in sc_last_error().  The first call
 * on each device looks up the array's device address (cudaGetSymbolAddress);
 * make that first call before any stream capture.  All calls share the array:
 * calls that overlap on the GPU (different streams, without ordering) race.
 * A bounded wait that expires in any call is recorded in the array's status
 * word, which keeps it until sc_layer_noalloc_status() reads it.
 */
int sc_layer_forward_noalloc(const sc_layer_args* args, void* stream);

/* Synchronises `stream`, returns SC_ERR_TIMEOUT if a bounded wait expired in a
 * sc_layer_forward_noalloc call on the current device since the last query
 * (else SC_OK, or SC_ERR_CUDA), and clears the word.  Allocates nothing. */
int sc_layer_noalloc_status(void* stream);

/* Test hook of the failure path; not for production use.  While ns > 0, the
 * first MMA-issuing thread of every CTA of the per-layer attention kernel
 * (sc_layer_forward, sc_layer_forward_noalloc and the per-layer part of the
 * stacks) first waits at most ns nanoseconds on a barrier that nothing
 * completes.  That bounded wait expires: the CTA abandons its work, drains
 * its copies and matrix products, frees its tensor memory and records
 * SC_ERR_TIMEOUT in the status word, so the call's results are undefined and
 * the status query reports SC_ERR_TIMEOUT.  ns = 0 (the default) turns it off.
 * Process-wide; read when a call enqueues its kernels. */
void sc_debug_stall_waits(unsigned long long ns);

/* Test hook of the graph route of eager stack calls (sc_stack_forward,
 * sc_stack_forward_host): since the library was loaded, how many calls were
 * recorded into a new graph (*recorded) and how many launched a kept graph
 * (*reused).  Process-wide; either pointer may be NULL. */
void sc_debug_graph_counts(unsigned long long* recorded, unsigned long long* reused);

/* Bytes of workspace a call with these sizes needs (0 on invalid sizes). */
size_t sc_workspace_size(int B, int L, int H);

/* One layer (Sec. "Sparse Attention" + Sec. "Token Pruning").  Errors: see sc_status. */
int sc_layer_forward(const sc_layer_args* args, void* workspace, size_t workspace_bytes,
                     void* stream);

/* The pruned stack (Fig. "sparsecoder": sparse attention with layer-wise
 * token pruning, 12 layers in the paper's encoder).  Errors: see sc_status.
 *
 * Execution: a sequence runs layer by layer through the per-layer kernels
 * while it has more than SC_TAIL_MAX_LEN current tokens; from the first layer at
 * which it has at most SC_TAIL_MAX_LEN (after padding removal or after a layer's
 * pruning) its
 * remaining layers run in one cluster kernel launched once at the end of the
 * call (one thread-block cluster of H CTAs per sequence, when the device can
 * schedule clusters of H <= 16 CTAs and n_layers <= 64).  The hand-over is
 * decided on the device: the call never waits for the GPU and can be captured
 * in a CUDA graph.  Results are the same function of the inputs either way
 * (within the stated tolerances).
 *
 * Launches: in a CUDA graph (a call made while `stream` is being captured)
 * the per-layer kernels run in a loop whose condition the device sets, so
 * the layers that every sequence runs in the cluster kernel launch nothing.
 * An eager call (stream not capturing) that has both kinds of kernels in its
 * plan runs the same way: the library records the call into a graph of its
 * own, keeps the instantiated graph (up to 16 per process, least recently
 * used replaced first) and launches it on `stream`; a later call with the
 * same arguments (sizes, device addresses, the alpha and global values, the
 * workspace, the device, and the process-wide settings read at enqueue)
 * launches the kept graph without recording again.  Recording and
 * instantiating make the first call with new arguments cost more host time
 * (a fraction of a millisecond).  With SC_STACK_PLAIN_LAUNCHES, or when the
 * plan has only one kind of kernel, an eager call launches its kernels
 * directly: every layer's per-layer kernels, which skip the sequences that
 * the cluster kernel runs. */
int sc_stack_forward(const sc_stack_args* args, void* workspace, size_t workspace_bytes,
                     void* stream);

/* sc_stack_forward, plus CUDA events (cudaEvent_t passed as void*) recorded on
 * `stream` around the kernels, for timing on the launching stream:
 * events[0] before the first launch, events[1] after the padding-removal
 * kernel, then for layer l: events[2+3l] after its rows kernel, events[3+3l]
 * after its cols kernel (scores, threshold, compaction) and events[4+3l] after
 * the gather of the next layer's rows, and events[2+3*n_layers] after the
 * cluster kernel of the short sequences.  Events of kernels that a call does
 * not launch are recorded anyway (back to back).  n_events >= 3 + 3 * n_layers.
 * A NULL entry records nothing at that point, so that kernels on both sides of
 * it stay chained (programmatic dependent launch) as in an uninstrumented call,
 * e.g. events[2] = NULL times layer 0's rows and cols kernels together as they
 * overlap.  The events are caller-owned. */
int sc_stack_forward_profiled(const sc_stack_args* args, void* workspace, size_t workspace_bytes,
                              void* stream, void** events, int n_events);

/* Number of kernels that sc_stack_forward launches for these arguments (on the
 * current device) when it launches them directly (SC_STACK_PLAIN_LAUNCHES, or
 * a plan with one kind of kernel), in *count.  A call that runs as a graph
 * launches prep, [padding-removal gather], then rows, cols, gather and a
 * loop-advance kernel for layer 0 and for each later layer that some sequence
 * still runs per layer, then the cluster kernel.  Only the sizes, n_layers,
 * flags, pad_mask (NULL or not) and the global list are read; no pointer is
 * dereferenced and nothing is launched.  Errors: see sc_status (SC_ERR_CUDA
 * without a usable device). */
int sc_stack_launch_count(const sc_stack_args* args, int* count);

/*
 * The pruned stack with its inputs and results in HOST memory: the same
 * computation and results as sc_stack_forward (Fig. "sparsecoder"; Sec.
 * "Sparse Attention", "Token Pruning"), for callers whose tensors live on the
 * host.  The kernels move only what the method uses: layer l reads, over the
 * host link, the Q/K/V rows of the tokens that survived layers 0..l-1 (token
 * pruning, Sec. "Token Pruning" Step 3, removes the others from every later
 * layer), and the results are written back only where sc_stack_forward
 * defines them.
 *
 * args       as for sc_stack_forward, except that Q, K, V, pad_mask (or NULL),
 *            O, scores, pos and len are HOST pointers to page-locked memory
 *            (cudaHostAlloc / cudaMallocHost, or cudaHostRegister'ed) that the
 *            device can address; alpha and global_pos are host arrays as there.
 *            Written on the host: len (all of it), and for every (l, b) the
 *            first len[l][b] entries of pos[l][b] (l <= n_layers), scores[l][b]
 *            and rows of O[l][b] (l < n_layers); every other entry is left as
 *            it was.
 * workspace  DEVICE memory of sc_stack_host_workspace_size(n_layers, B, L, H)
 *            bytes (256-byte aligned): the scratch of sc_stack_forward followed
 *            by device copies of the results of the layers that run on the
 *            per-layer kernels (the cluster kernel writes the results of the
 *            layers it runs to the host buffers directly).
 *
 * Asynchronous on `stream` like every call: the host buffers must stay
 * allocated and unmodified (inputs) or unread (results) until the stream has
 * passed the call.  Capturable in a CUDA graph (it issues kernels only); an
 * eager call runs through a kept graph of the library (the export included)
 * under the same rules as sc_stack_forward, the mapped host addresses being
 * part of its key.
 * Errors: as sc_stack_forward, and SC_ERR_INVALID_ARG with nothing launched
 * when a host range is not page-locked memory mapped for the device (checked
 * at both ends of each range) or a mapped address is misaligned (Q, K, V, O:
 * 16 bytes; scores, pos, len: 4 bytes).
 */
size_t sc_stack_host_workspace_size(int n_layers, int B, int L, int H);
int sc_stack_forward_host(const sc_stack_args* args, void* workspace, size_t workspace_bytes,
                          void* stream);

/* Number of kernels that sc_stack_forward_host launches for these arguments,
 * as sc_stack_launch_count for sc_stack_forward. */
int sc_stack_host_launch_count(const sc_stack_args* args, int* count);

/*
 * The per-layer attention for windows of at most 256 tokens on each side can
 * run in one of two designs (process-wide, read when a call enqueues its
 * kernels; both give the method's results within the stated tolerances):
 *   SC_ROWS_TWO_PASS (default): the row pass keeps only O and each row's LSE;
 *     a second pass over the band recomputes S^T and its exponentials to form
 *     the column sums of Sec. "Pruning" ("accumulated vertically", Fig. 1) in
 *     fp32.
 *   SC_ROWS_SINGLE_PASS: every band tile's S = q.k/8 is computed and
 *     exponentiated once; each tile's bf16 probabilities stay on chip until
 *     the row's normaliser is known, and the column sums are then one
 *     tensor-core product per tile (P~^T times the per-row weights
 *     2^(m_t - LSE_i)).  The bf16 rounding of P~ bounds the relative error of
 *     each score by 2^-9; sequences of at least a few hundred tokens stay well
 *     inside 1e-5 absolute, sequences of a few dozen tokens may not.
 * Wider windows always use the two-pass design.  Returns SC_ERR_INVALID_ARG
 * for any other value.
 */
#define SC_ROWS_SINGLE_PASS 0
#define SC_ROWS_TWO_PASS 1
int sc_select_rows_kernel(int which);

/* Synchronises `stream`, returns SC_ERR_TIMEOUT if any kernel since the last
 * query recorded an expired wait (else SC_OK, or SC_ERR_CUDA), and clears
 * the status word. */
int sc_workspace_status(void* workspace, size_t workspace_bytes, void* stream);

/*
 * The encoder layer around the path (the steps either side of the attention,
 * Fig. "sparsecoder"): a RoBERTa-style post-LN layer whose
 * self-attention is the sparse attention with token pruning above, and whose
 * output projection and feed-forward block run on the kept tokens only.  D = 64 H.
 *
 *   Q, K, V = X W_qkv^T + b_qkv            (W_qkv rows: the D outputs of Q, then K, then V)
 *   O, s, keep = sc_layer_forward(Q, K, V)
 *   S1 = X[kept] + O[kept] W_o^T + b_o;  H1 = LN1(S1)
 *   Y  = LN2(H1 + GELU(H1 W_1^T + b_1) W_2^T + b_2)
 * LN(x) = (x - mean) / sqrt(var + 1e-5) * gamma + beta over the D features
 * (population variance); GELU(x) = x/2 (1 + erf(x / sqrt 2)).  Stored as bf16:
 * Q, K, V, O, H1, GELU's output, Y; S1 and the second sum stay fp32.
 * Kernels per call: the Q/K/V GEMM, the attention layer's kernels, a copy of
 * O's kept rows into consecutive rows, the output-projection GEMM (X[kept]
 * gathered in its epilogue), layer norm, the two feed-forward GEMMs, layer norm.
 *
 * X          bf16 [B][L][D] hidden states in current order (row c of sequence b
 *            is current token c; rows at or beyond len[b] are never read).
 * len, pos, w, global_pos, n_global, keep_rule, alpha, theta: as sc_layer_args.
 * W_qkv bf16 [3D][D], b_qkv fp32 [3D]; W_o bf16 [D][D], b_o [D];
 * ln1_gamma, ln1_beta fp32 [D]; W_1 bf16 [4D][D], b_1 [4D]; W_2 bf16 [D][4D],
 * b_2 [D]; ln2_gamma, ln2_beta [D].  Weights are [out][in] (row per output).
 * Y          bf16 [B][L][D] out: the kept tokens' outputs, compacted (row k of
 *            sequence b is its k-th kept token): the next layer's X, with
 *            len_out and pos_out as its len and pos.
 * O          bf16 [B][L][D] out: the attention output of every current token.
 * scores, pos_out, len_out: as sc_layer_args.
 * H must be even (D a multiple of 128) and at most 16.
 */
typedef struct {
  int B, L, H, w;
  const uint16_t* X;
  const int32_t* len;
  const int32_t* pos;
  const int32_t* global_pos;
  int n_global;
  int keep_rule;
  float alpha;
  const float* theta;
  const uint16_t* W_qkv;
  const float* b_qkv;
  const uint16_t* W_o;
  const float* b_o;
  const float* ln1_gamma;
  const float* ln1_beta;
  const uint16_t* W_1;
  const float* b_1;
  const uint16_t* W_2;
  const float* b_2;
  const float* ln2_gamma;
  const float* ln2_beta;
  uint16_t* Y;
  uint16_t* O;
  float* scores;
  int32_t* pos_out;
  int32_t* len_out;
} sc_encoder_args;

/* Bytes of workspace sc_encoder_layer_forward needs (0 on invalid sizes). */
size_t sc_encoder_workspace_size(int B, int L, int H);

/* One encoder layer (see sc_encoder_args).  Errors: see sc_status. */
int sc_encoder_layer_forward(const sc_encoder_args* args, void* workspace,
                             size_t workspace_bytes, void* stream);

/*
 * The GEMM of the encoder layer on its own: for every sequence b and row
 * r < rows[b] (rows == NULL: all L rows),
 *   out[b L + r][n] = act(sum_k A[b L + g(r)][k] W[n][k] + bias[n]) (+ res[...][n])
 * with g(r) = gidx[b L + r] (gidx == NULL: r), act = GELU when gelu != 0, and
 * res (bf16, NULL for none) read at row b L + g(r) when res_gathered, else at
 * b L + r.  A bf16 [B L][K], W bf16 [N][K] ([out][in]), bias fp32 [N] or NULL,
 * out [B L][N] bf16, or fp32 when out_f32.  N % 128 == 0, K % 64 == 0, K <= 8192;
 * A and W 16-byte aligned.  `workspace` (>= 256 bytes, 256-byte aligned) holds
 * the status word read by sc_workspace_status.
 */
typedef struct {
  int B, L, N, K;
  const uint16_t* A;
  const int32_t* rows;
  const int32_t* gidx;
  const uint16_t* W;
  const float* bias;
  int gelu;
  const uint16_t* res;
  int res_gathered;
  void* out;
  int out_f32;
} sc_linear_args;

int sc_linear_forward(const sc_linear_args* args, void* workspace, size_t workspace_bytes,
                      void* stream);

/* Layer norm of the rows (b, r), r < rows[b] (rows == NULL: all): in fp32
 * [B L][D], out bf16 [B L][D], gamma/beta fp32 [D], eps as given; D % 32 == 0,
 * D <= 1024. */
int sc_layer_norm_forward(int B, int L, int D, const int32_t* rows, const float* in,
                          const float* gamma, const float* beta, float eps, uint16_t* out,
                          void* stream);

/* Static, human-readable name of a status code. */
const char* sc_status_string(int status);

/* Detail of the most recent SC_ERR_CUDA on the calling thread (which step
 * failed and the CUDA error text); an empty string if none.  Valid until the
 * next call on this thread. */
const char* sc_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* SPARSECODER_H */
