/*
 * ordermoe.h - C ABI of the GB300 (sm_103a) OrderMoE hot-path library.
 *
 * The library computes one MoE layer forward with similarity-aware expert
 * substitution, after "OrderMoE: an expert similarity driven distributed edge
 * MoE inference" (arXiv 2607.17154), plus the offline similarity, grouping and
 * placement that feed it. Edge servers are a logical expert-to-server
 * placement map on one GPU: no data moves between servers.
 *
 * Conventions for every call below:
 *  - Pointers are DEVICE pointers owned by the caller unless a parameter says
 *    "host". The library keeps no pointer after a call returns.
 *  - bf16 tensors are passed as uint16_t bit patterns, row-major, dense.
 *  - Every call only enqueues work on `stream` (NULL = the legacy default
 *    stream) and returns; nothing is synchronised and nothing is read back to
 *    the host, except where a call says so.
 *  - Return value: ORDERMOE_OK, or an error code; ordermoe_last_error() then
 *    gives a message (thread-local). Argument errors are detected on the host
 *    before anything is enqueued. Errors found by a kernel (an index out of
 *    range, a NaN logit, a bounded wait that ran out) set a device error word
 *    that ordermoe_device_error() reads.
 *  - Limits: E <= 64 experts, M <= 32 servers, k <= 8 slots per token.
 */
#ifndef ORDERMOE_H
#define ORDERMOE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t / CUstream. */
typedef struct CUstream_st* ordermoe_stream_t;

enum {
  ORDERMOE_OK = 0,
  ORDERMOE_ERR_INVALID_ARG = 1,       /* null pointer, bad size, bad alignment  */
  ORDERMOE_ERR_UNSUPPORTED_SHAPE = 2, /* outside the limits stated per call      */
  ORDERMOE_ERR_CAPACITY = 3,          /* placement: sum C_m < sum p, or overflow */
  ORDERMOE_ERR_CUDA = 4,              /* a CUDA runtime/driver call failed       */
  ORDERMOE_ERR_DEVICE_CHECK = 5       /* a kernel reported an error (see below)  */
};

/* Device error word values (ordermoe_device_error). */
enum {
  ORDERMOE_DEV_OK = 0,
  ORDERMOE_DEV_NAN_LOGIT = 1,     /* route_select: a logit was NaN             */
  ORDERMOE_DEV_BAD_INDEX = 2,     /* an expert/server index out of range       */
  ORDERMOE_DEV_NO_CANDIDATE = 3,  /* selection: target expert placed nowhere   */
  ORDERMOE_DEV_WAIT_TIMEOUT = 4,  /* a bounded pipeline wait ran out           */
  ORDERMOE_DEV_BAD_VALUE = 5      /* a memory demand p or a reference delay <= 0 */
};

#define ORDERMOE_MAX_EXPERTS 64
#define ORDERMOE_MAX_SERVERS 32
#define ORDERMOE_MAX_TOPK 8

/* Message for the last error returned on this host thread. */
const char* ordermoe_last_error(void);

/* Library version, major * 10000 + minor * 100 + patch. */
int ordermoe_version(void);

/* Reads and clears the device error word of the current device. This call
 * synchronises the device. *code (host) receives an ORDERMOE_DEV_* value and
 * *detail (host, nullable) a kernel-specific detail (e.g. the token index).
 * Returns ORDERMOE_ERR_DEVICE_CHECK when *code != 0, else ORDERMOE_OK. */
int ordermoe_device_error(int* code, int* detail);

/* Sets the limit, in nanoseconds, of every bounded device-side wait in kernels
 * launched afterwards on this host thread (default 2e9 = 2 s). A wait that runs
 * out sets ORDERMOE_DEV_WAIT_TIMEOUT and the kernel returns early. */
int ordermoe_set_wait_limit_ns(uint64_t limit_ns);

/* Launches one kernel whose single bounded wait is on an mbarrier that nothing
 * arrives at, so that the wait runs out after `limit_ns`. Used to test that
 * bounded waits end and report ORDERMOE_DEV_WAIT_TIMEOUT. */
int ordermoe_selftest_wait_timeout(uint64_t limit_ns, ordermoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Per-layer selection tables.
 *
 * A device buffer of ordermoe_tables_bytes(E, M) bytes, written by
 * ordermoe_build_tables and read by ordermoe_route_select. Layout (byte
 * offsets; all little-endian):
 *     0  int32  magic 0x4f4d5442, E, M, reserved
 *    16  float  theta, qbar
 *    64  uint32 pmask[64]   bit m set <=> x_{m,e} = 1          (placement)
 *   320  uint64 subst[64]   bit k set <=> e_k in R_{l,e} (Eq. 7)
 *   832  float  Qtab[E][E]  Q_l(r,k) of Eq. 18, phi = identity
 *        float  Cq[E][E]    omega_Q Q_l(r,k) / Qbar (quality term of Eq. 38)
 *        float  A[M][M][M]  A[a][s][m] = omega_T d(s,m) / d_ref(a) (delay term
 *                           of Eq. 38; d of Eq. 37; d_ref(a) = c / F_a)
 * ------------------------------------------------------------------------ */
size_t ordermoe_tables_bytes(int E, int M);

/* Builds the selection tables of one layer (Sections III-B, III-D, III-E and
 * V-A: Eqs. 7, 18, 37, 38).
 *   sim        [E][E] f32   expert similarity Sim_l (Eq. 4)
 *   group      [E] i32      similarity group of each expert (Eq. 26)
 *   placement  [M][E] u8    x_{m,l,e} (1 = expert e deployed on server m)
 *   theta      similarity threshold theta_l of the layer (Eq. 6 / Eq. 7)
 *   qbar       per-token quality budget Qbar (Eq. 39), >= 0
 *   F [M], B [M][M], tau [M][M]  f64: server compute (flop/s), link bandwidth
 *              (bytes/s) and latency (s); the diagonals are not read
 *   z          bytes moved when a token changes server (z_l of Eq. 37)
 *   c          flop of one expert on one token (c_l of Eq. 15)
 *   omega_T, omega_Q  cost weights of Eq. 38
 *   tables     out, device buffer of tables_bytes >= ordermoe_tables_bytes(E,M)
 * fp64 terms are computed with correctly rounded IEEE operations (no fused
 * multiply-add) and rounded once to fp32. */
int ordermoe_build_tables(const float* sim, const int32_t* group, const uint8_t* placement,
                          int E, int M, float theta, float qbar, const double* F, const double* B,
                          const double* tau, double z, double c, double omega_T, double omega_Q,
                          void* tables, size_t tables_bytes, ordermoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Router + softmax + top-k + server-expert selection (Alg. 2 with horizon
 * H = 1, Section V; the router output is the "target expert from the local
 * router" of Alg. 2).
 *   X          [T][d] bf16  token representations (ignored if logits_in)
 *   W_r        [E][d] bf16  router weights (ignored if logits_in)
 *   logits_in  [T][E] f32, nullable: when given, the router GEMM is skipped
 *              and these logits are used
 *   renorm     1: top-k gate weights renormalised to sum to 1 over the k slots
 *   tables     the layer's tables (ordermoe_build_tables)
 *   home       [T] u8   home (access) server a(i) of each token
 *   loc        [T] u8   in/out: server holding the token before / after the
 *              layer (Eq. 36, Eq. 44); set loc = home before the first layer
 *   qhat       [T] f32  in/out: accumulated quality loss (Eq. 44); 0 at start
 *              loc and qhat may both be NULL: every token then starts at its
 *              home server with zero loss (the first layer) and the new state
 *              is not written
 *   logits_out [T][E] f32, nullable: the router logits
 *   topk_idx   [T][k] i32  routed (target) experts, rank order: by logit,
 *              equal logits to the lower expert index
 *   topk_w     [T][k] f32  gate weights of the routed slots (fp32 softmax
 *              over all E logits, the terms summed in expert order)
 *   chosen_expert [T][k] i32  executed expert k* per slot (Eq. 43)
 *   chosen_server [T][k] u8   executing server m* per slot
 *   kind       [T][k] u8   0 local exact, 1 local substitute, 2 remote exact,
 *              3 remote substitute (Section VI-C's execution types)
 *   counters   [4] i32, nullable: += number of slots of each kind
 * Readings of the paper: with k > 1 the selection runs per slot in rank
 * order; a substitute is never one of the token's routed experts nor a
 * substitute already given to it; the token's new location is the server of
 * slot 0; ties in Eq. 43 go to lower cost, exact, current server, lower
 * server, lower expert. Shapes: 1 <= E <= 64, 1 <= k <= min(E, 8),
 * d % 64 == 0 (X and W_r 16-byte aligned) unless logits_in is given.
 * A token with a NaN logit sets ORDERMOE_DEV_NAN_LOGIT (detail: the token);
 * its topk_idx row is -1 and its topk_w row 0; its chosen_expert,
 * chosen_server, kind, loc and qhat are not written. */
int ordermoe_route_select(const uint16_t* X, const uint16_t* W_r, const float* logits_in, int T,
                          int E, int d, int k, int renorm, const void* tables, size_t tables_bytes,
                          const uint8_t* home, uint8_t* loc, float* qhat, float* logits_out,
                          int32_t* topk_idx, float* topk_w, int32_t* chosen_expert,
                          uint8_t* chosen_server, uint8_t* kind, int32_t* counters,
                          ordermoe_stream_t stream);

/* Alg. 2 with look-ahead horizon H (Eqs. 41-43): as ordermoe_route_select,
 * but each candidate (m, k) of this layer costs g_l(m, k) + Phi^(H-1)(m, k),
 * the expected cheapest cost of the next H - 1 layers from server m:
 *   Phi^(h)(m, k) = sum_{k'} P_l(k -> k') min over the feasible (m', k'') of
 *                   target k' at layer l + 1 (from server m, with the loss
 *                   accumulated so far) of g_{l+1}(m', k'') + Phi^(h-1)(m', k'')
 * (Eq. 42 read with the bracket closing after the per-step cost; future layers
 * have a single target and no distinct-expert rule).
 *   tables      H consecutive layer tables (this layer first), tables_stride
 *               bytes apart (a multiple of 16, >= ordermoe_tables_bytes(E, M))
 *   H           1..4 (1 gives exactly ordermoe_route_select's result)
 *   P           [H-1][E][E] f32: P_l .. P_{l+H-2} (ordermoe_transitions)
 * Every product and sum of Phi is one rounded fp32 operation, next targets in
 * ascending order, so decisions are reproducible bit for bit. */
int ordermoe_route_select_lookahead(const uint16_t* X, const uint16_t* W_r, const float* logits_in,
                                    int T, int E, int d, int k, int renorm, const void* tables,
                                    size_t tables_stride, int H, const float* P,
                                    const uint8_t* home, uint8_t* loc, float* qhat,
                                    float* logits_out, int32_t* topk_idx, float* topk_w,
                                    int32_t* chosen_expert, uint8_t* chosen_server, uint8_t* kind,
                                    int32_t* counters, ordermoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Token permutation: histogram + prefix sum + stable scatter of the T*k
 * (token, slot) entries by executed expert, and the row gather of X into
 * expert-contiguous order (the grouped layout the expert FFN consumes).
 *   chosen_expert [T][k] i32 (0 <= e < E)
 *   X          [T][d] bf16
 *   offsets    [E+1] i32 out: rows of expert e are offsets[e] .. offsets[e+1]-1
 *   row_token  [T*k] i32 out: token of each permuted row
 *   row_of     [T][k] i32 out: permuted row of each (token, slot)
 *   X_perm     [T*k][d] bf16 out: X_perm[row] = X[row_token[row]]
 *   workspace  device scratch of ordermoe_dispatch_workspace_bytes(T,k,E) bytes
 * Within one expert, rows keep the flat (t*k + j) order: the result is
 * unique. d % 8 == 0 and 16-byte aligned X / X_perm. */
size_t ordermoe_dispatch_workspace_bytes(int T, int k, int E);
int ordermoe_dispatch(const int32_t* chosen_expert, const uint16_t* X, int T, int k, int E, int d,
                      int32_t* offsets, int32_t* row_token, int32_t* row_of, uint16_t* X_perm,
                      void* workspace, size_t workspace_bytes, ordermoe_stream_t stream);

/* The permutation of ordermoe_dispatch, same arguments and results, for
 * callers that cannot give the library device memory: a plugin whose host
 * framework owns every device allocation through its own pool, or a serving
 * loop that may not call cudaMalloc once it runs. (The paper has no
 * counterpart; it is an interface convenience.) Its scratch is a fixed
 * 256 KB device array inside the library, present on every GPU that loads the
 * library until the process exits, so T*k is limited to 262144 entries
 * (larger calls fail with ORDERMOE_ERR_UNSUPPORTED_SHAPE). The array's device
 * address is looked up on the first call made on each device: make that
 * first call before any stream capture. The address is kept until the
 * process exits; after cudaDeviceReset of a device it is stale, so do not
 * call this entry point on a device the process has reset. All calls share the array, so calls
 * that overlap on the GPU (other streams, other host threads) race; nothing
 * in it needs clearing between calls. The call allocates nothing. */
int ordermoe_dispatch_noalloc(const int32_t* chosen_expert, const uint16_t* X, int T, int k,
                              int E, int d, int32_t* offsets, int32_t* row_token, int32_t* row_of,
                              uint16_t* X_perm, ordermoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Grouped SwiGLU expert FFN over the permuted rows (the Mixtral-style experts
 * of Section VI-A):
 *   H[row] = bf16( silu(x W1_e^T) * (x W3_e^T) ),  Y_perm[row] = bf16( H[row] W2_e^T )
 * for every row of expert e (offsets from ordermoe_dispatch, read on the
 * device: no host synchronisation). fp32 accumulation on tcgen05 tensor cores.
 *   X_perm [R][d] bf16, offsets [E+1] i32 (offsets[E] == R)
 *   W1, W3 [E][dff][d] bf16;  W2 [E][d][dff] bf16
 *   H      [R][dff] bf16 out (the SwiGLU activations; caller-owned scratch)
 *   Y_perm [R][d] bf16 out
 * Shapes: d % 256 == 0, dff % 128 == 0, all pointers 16-byte aligned. */
int ordermoe_expert_ffn(const uint16_t* X_perm, const int32_t* offsets, int R, const uint16_t* W1,
                        const uint16_t* W3, const uint16_t* W2, int E, int d, int dff, uint16_t* H,
                        uint16_t* Y_perm, ordermoe_stream_t stream);

/* The two halves of ordermoe_expert_ffn as separate launches (same shapes,
 * same rules): H = SwiGLU(X_perm W1^T, X_perm W3^T), then Y_perm = H W2^T. */
int ordermoe_expert_gate_up(const uint16_t* X_perm, const int32_t* offsets, int R,
                            const uint16_t* W1, const uint16_t* W3, int E, int d, int dff,
                            uint16_t* H, ordermoe_stream_t stream);
int ordermoe_expert_down(const uint16_t* H, const int32_t* offsets, int R, const uint16_t* W2,
                         int E, int d, int dff, uint16_t* Y_perm, ordermoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Weighted combine: y[t] = bf16( sum_{j=0..k-1} topk_w[t][j] * Y_perm[row_of[t][j]] )
 * with fp32 accumulation in slot order.
 *   Y_perm [T*k][d] bf16, row_of [T][k] i32, topk_w [T][k] f32, y [T][d] bf16 out.
 * d % 8 == 0, 16-byte aligned Y_perm / y. */
int ordermoe_combine(const uint16_t* Y_perm, const int32_t* row_of, const float* topk_w, int T,
                     int k, int d, uint16_t* y, ordermoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Residual map between stacked MoE layers (a decoder block without its
 * attention half; the paper's Mixtral-8x7B model, Section VI-A, stacks 32
 * such layers). The residual stream h (bf16) carries the layer outputs and
 * each layer reads its RMS-normalised copy x (pre-norm, unit gain):
 *   x_0 = RMSNorm(h_0),  h_{l+1} = h_l + y_l,  x_{l+1} = RMSNorm(h_{l+1}),
 *   RMSNorm(v)[c] = bf16( v[c] / sqrt(mean_c(v[c]^2) + eps) ).
 * Without the normalisation the outputs of random-weight SwiGLU experts grow
 * quadratically with their input and overflow within a few layers.
 *
 * ordermoe_rmsnorm: x = RMSNorm(h) for T rows of d.
 *   h, x [T][d] bf16 (16-byte aligned), eps > 0; x may not overlap h.
 * ordermoe_combine_residual_norm: the weighted combine added to the residual
 * stream, and the next layer's input, in one pass:
 *   h_out[t] = bf16( h[t] + sum_{j<k} topk_w[t][j] Y_perm[row_of[t][j]] )
 *   (fp32, slot order), x_out[t] = RMSNorm(h_out[t]) (sum of squares of the
 *   bf16 values of h_out in fp32, fixed reduction order).
 *   Y_perm [T*k][d], h, h_out, x_out [T][d] bf16 (16-byte aligned, h, h_out
 *   and x_out mutually disjoint); row_of, topk_w as ordermoe_combine; d % 8 == 0.
 *   A row_of entry outside [0, T*k) sets ORDERMOE_DEV_BAD_INDEX (detail: the
 *   token) and leaves that token's h_out and x_out unwritten. */
int ordermoe_rmsnorm(const uint16_t* h, int T, int d, float eps, uint16_t* x,
                     ordermoe_stream_t stream);
int ordermoe_combine_residual_norm(const uint16_t* Y_perm, const int32_t* row_of,
                                   const float* topk_w, const uint16_t* h, int T, int k, int d,
                                   float eps, uint16_t* h_out, uint16_t* x_out,
                                   ordermoe_stream_t stream);

/* ------------------------------------------------------------------------
 * One whole MoE layer: route_select, dispatch, expert_gate_up, expert_down and
 * combine in order on `stream`, with all intermediates in `scratch`.
 * The descriptor (host memory) holds device pointers owned by the caller:
 *   W_r [E][d], W1/W3 [E][dff][d], W2 [E][d][dff] bf16; tables of the layer;
 *   scratch: ordermoe_layer_scratch_bytes(T_max, E, d, dff, k) bytes,
 *   256-byte aligned. */
typedef struct {
  int T_max, E, d, dff, k, renorm;
  const uint16_t* W_r;
  const uint16_t* W1;
  const uint16_t* W3;
  const uint16_t* W2;
  const void* tables;
  size_t tables_bytes;
  void* scratch;
  size_t scratch_bytes;
  /* look-ahead (Eqs. 41-43); lookahead_H <= 1 selects myopically. With H > 1
   * `tables` must be followed by the next H - 1 layers' tables at
   * tables_stride bytes, and P holds [H-1][E][E] transition matrices. */
  int lookahead_H;
  size_t tables_stride;
  const float* P;
} ordermoe_layer_desc;

size_t ordermoe_layer_scratch_bytes(int T_max, int E, int d, int dff, int k);

/* y[t] = MoE layer output of token t, t < T <= T_max.
 *   X [T][d] bf16, home [T] u8, y [T][d] bf16 out.
 *   loc [T] u8 and qhat [T] f32 in/out (Eq. 36 / Eq. 44), or both NULL: the
 *   tokens then start at their home server with zero accumulated loss (the
 *   first MoE layer) and the new state is not returned.
 *   counters [4] i32 device, nullable (see ordermoe_route_select).
 *   host_io = 0: X, home, loc, qhat, y are device pointers.
 *   host_io = 1: they are HOST pointers (pinned for asynchronous copies); the
 *   call enqueues the host -> device copies, the layer, and the device -> host
 *   copies on `stream`; the caller synchronises before reading y.
 * Shapes as ordermoe_route_select and ordermoe_expert_ffn. */
int ordermoe_layer_forward(const ordermoe_layer_desc* layer, int T, const uint16_t* X,
                           const uint8_t* home, uint8_t* loc, float* qhat, uint16_t* y,
                           int32_t* counters, int host_io, ordermoe_stream_t stream);

/* One layer of a stack on the residual map above (device pointers only):
 * the layer routes and runs x (= RMSNorm(h)), then
 * ordermoe_combine_residual_norm writes h_out = h + y and x_out =
 * RMSNorm(h_out), the next layer's h and x. loc / qhat, counters and the
 * look-ahead fields of the descriptor as ordermoe_layer_forward; logits_out
 * [T][E] f32 (nullable) receives the router logits of x (the calibration
 * pass of a stack records them for ordermoe_transitions_strided).
 *   x, h, h_out, x_out [T][d] bf16, 16-byte aligned, h / h_out / x_out
 *   mutually disjoint; eps > 0. */
int ordermoe_layer_forward_residual(const ordermoe_layer_desc* layer, int T, const uint16_t* x,
                                    const uint16_t* h, const uint8_t* home, uint8_t* loc,
                                    float* qhat, float eps, uint16_t* h_out, uint16_t* x_out,
                                    float* logits_out, int32_t* counters, ordermoe_stream_t stream);

/* nbatch independent batches of T tokens through one layer, from and to
 * pinned HOST memory, each batch as ordermoe_layer_forward with host_io = 1
 * and the tokens at their home servers (a first layer: no loc / qhat), with
 * the copies overlapped with the compute: batch b's inputs are copied in
 * while batch b - 1 computes, and its output is copied out while batch b + 1
 * computes (two staging slots, two copy streams owned by the library, one per
 * device). Serves a queue of requests; has no counterpart in the paper.
 *   X [nbatch][T][d] bf16, home [nbatch][T] u8, y [nbatch][T][d] bf16 out
 *   (host); counters as ordermoe_layer_forward.
 *   layer->scratch: ordermoe_layer_batches_scratch_bytes(T_max, E, d, dff, k)
 *   bytes (the layer scratch plus a second staging slot).
 * The call enqueues everything; `stream` is ordered after every copy (also
 * when it returns an error after enqueueing some), so the caller synchronises
 * it before reading y. Calls on the same device from several host threads are
 * enqueued one at a time (the copy streams are the device's); each needs its
 * own layer->scratch. */
size_t ordermoe_layer_batches_scratch_bytes(int T_max, int E, int d, int dff, int k);
int ordermoe_layer_forward_batches(const ordermoe_layer_desc* layer, int nbatch, int T,
                                   const uint16_t* X, const uint8_t* home, uint16_t* y,
                                   int32_t* counters, ordermoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Offline expert similarity (Section III-B, Eqs. 3-5; Alg. 1).
 * For each layer l: H_l = W_r^l X_cal^T (router logits over the calibration
 * tokens, fp32 accumulation on tcgen05 tensor cores),
 * Sim_l(i,j) = <H_l,i, H_l,j> / (|H_l,i| |H_l,j|) (Eq. 4; diagonal exactly 1,
 * 0 for a zero-norm row), and the activation counts n_l^j = number of
 * calibration tokens whose top-k_freq experts include j (Eq. 5; ties to the
 * lower index).
 *   W_r      [L][E][d] bf16 (the L router matrices stacked)
 *   X_cal    [N][d] bf16 calibration tokens
 *   sim      [L][E][E] f32 out;  counts [L][E] i32 out
 *   workspace  device scratch of ordermoe_similarity_workspace_bytes(L,E,N)
 *              bytes, 256-byte aligned (holds H in fp32 and partial Grams)
 * Shapes: d % 64 == 0, 1 <= k_freq <= E <= 64, 1 <= N <= 65535 * 1024, L <=
 * 65535. Gram partial sums are reduced in a fixed order: results are
 * deterministic. */
size_t ordermoe_similarity_workspace_bytes(int L, int E, int64_t N);
int ordermoe_similarity(const uint16_t* W_r, const uint16_t* X_cal, int L, int E, int d, int64_t N,
                        int k_freq, float* sim, int32_t* counts, void* workspace,
                        size_t workspace_bytes, ordermoe_stream_t stream);

/* After ordermoe_similarity returns (and until the workspace is reused), the
 * first N * L * E * 4 bytes of its workspace hold the calibration logits
 * H[n][l][e] in fp32, token-major: the input ordermoe_transitions takes. */

/* ordermoe_similarity without the calibration logits: the same arguments,
 * workspace size and results (sim and counts bit for bit), but the first
 * N * L * E * 4 bytes of the workspace are left undefined, which saves
 * writing them (1.6 GB for 24 layers x 64 experts x 262144 tokens) when no
 * ordermoe_transitions call follows. Where the tensor-core path does not apply
 * (E not in {8, 16, 32, 64}) the logits are computed and kept anyway. */
int ordermoe_similarity_no_logits(const uint16_t* W_r, const uint16_t* X_cal, int L, int E, int d,
                                  int64_t N, int k_freq, float* sim, int32_t* counts,
                                  void* workspace, size_t workspace_bytes,
                                  ordermoe_stream_t stream);

/* Expert transition statistics, Eq. 41, from calibration logits
 * [N][L][E] f32 (token-major, layer-stacked): n_l(k -> k') counts, for every
 * token, each pair (k in its top-k_freq at layer l, k' in its top-k_freq at
 * layer l + 1) -- the paper has one target per token; with top-k every routed
 * pair counts. P_l(k -> k') = n / sum_k'' n(k -> k'') (fp64, rounded once;
 * a row without transitions is 0).
 *   counts [L-1][E][E] i32 out, P [L-1][E][E] f32 out. Needs L >= 2. */
int ordermoe_transitions(const float* logits, int64_t N, int L, int E, int k_freq, int32_t* counts,
                         float* P, ordermoe_stream_t stream);

/* ordermoe_transitions over logits in any layout: the E logits of token n at
 * layer l start at logits + n * token_stride + l * layer_stride (floats; both
 * strides >= E). Layer-major logits [L][N][E], as a stack's calibration pass
 * records them one layer at a time, have token_stride = E and
 * layer_stride = N * E; ordermoe_transitions is token_stride = L * E,
 * layer_stride = E. Same results and rules. */
int ordermoe_transitions_strided(const float* logits, int64_t N, int L, int E, int k_freq,
                                 int64_t token_stride, int64_t layer_stride, int32_t* counts,
                                 float* P, ordermoe_stream_t stream);

/* Activation counts of Eq. 5 from given logits [N][E] f32 (top-k_freq per
 * token, ties to the lower index). counts [E] i32 out (overwritten). */
int ordermoe_expert_counts(const float* logits, int64_t N, int E, int k_freq, int32_t* counts,
                           ordermoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Grouping and mandatory placement (Section IV-A/B; Alg. 1), all
 * layers in order:
 *   theta_l = theta_min + (theta_max - theta_min)(L - l)/(L - 1), l = 1..L
 *            (Eq. 6; L == 1 uses theta_single);
 *   greedy representative cover (Eqs. 24-26): experts by decreasing count
 *            (ties: lower index) become a new dominant when their largest Sim
 *            to the existing dominants is < theta_l, else join the most similar
 *            dominant's group (ties: the earlier dominant); group id = the
 *            dominant's creation order;
 *   importance I = alpha_f f + alpha_r rho (Eqs. 27-28);
 *   placement (Eqs. 29-31): experts by (p desc, I desc, index asc), feasible
 *            servers b_m + p <= C_m, score lambda1 b_m / C_m + lambda2 eta
 *            (lambda1, lambda2 >= 0, p >= 0 and C_m > 0 finite; a negative
 *            or NaN p (detail = l * E + j), a negative or NaN score or a bad
 *            C_m sets ORDERMOE_DEV_BAD_VALUE),
 *            lowest score (ties: lower m); experts with no feasible server go,
 *            after the layer, to the server with the most free memory. The
 *            used memory b_m accumulates over the layers.
 *   sim [L][E][E] f32, counts [L][E] i32, p [L][E] f64 (memory of each
 *   expert), C [M] f64 (server capacities)
 *   group [L][E] i32 out, n_groups [L] i32 out, theta [L] f32 out,
 *   importance [L][E] f64 out (nullable; the input of ordermoe_replicate),
 *   placement [L][M][E] u8 out, used [M] f64 out,
 *   status [1] i32 out (device): ORDERMOE_OK, or ORDERMOE_ERR_CAPACITY when
 *   sum C < sum p or a waiting-list expert overflowed its server.
 *   workspace: device scratch of ordermoe_place_workspace_bytes(L, E) bytes
 *   (the per-layer placement orders between the per-layer pass, which runs
 *   the layers in parallel, and the placement pass, which runs them in order). */
size_t ordermoe_place_workspace_bytes(int L, int E);
int ordermoe_place(const float* sim, const int32_t* counts, int L, int E, int M, double theta_min,
                   double theta_max, double theta_single, double alpha_f, double alpha_r,
                   double lambda1, double lambda2, const double* p, const double* C,
                   int32_t* group, int32_t* n_groups, float* theta, double* importance,
                   uint8_t* placement, double* used, int32_t* status, void* workspace,
                   size_t workspace_bytes, ordermoe_stream_t stream);

/* Self-test of the quotient the placement's scores use (no counterpart in the
 * paper): out[i] = a[i] / b[i] rounded to nearest, computed as the placement
 * computes b_m / C_m (a reciprocal and Markstein's correction step).
 * a, b, out: [n] f64 device. For tests that compare it with IEEE division. */
int ordermoe_selftest_div_rn(const double* a, const double* b, double* out, int64_t n,
                             ordermoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Importance-aware redundant deployment (Section IV-C, Eqs. 32-35; Alg. 1),
 * after the mandatory placement, over all layers:
 *   y[m][l][g] = 1 when server m hosts an expert of group g of layer l (Eq. 32);
 *   benefit of a replica of expert j of layer l on server m:
 *     B = pi_m * I_l^j * (1 - y[m][l][g(j)]) / p_l^j          (Eq. 33);
 *   it fits when b_m + p_l^j <= C_m                          (Eq. 35);
 *   greedy (Eq. 34): deploy the largest fitting positive benefit (ties: lower
 *   layer, then lower server, then lower expert), update y and b_m, repeat
 *   until no fitting candidate has a positive benefit.
 * Memory and coverage are per server and a benefit only ever drops to 0, so
 * the greedy runs as one independent pass per server (one CTA each): its
 * candidates sorted by (benefit desc, layer, expert), then swept in order.
 *   group [L][E] i32 (ids < E), importance [L][E] f64 (ordermoe_place's),
 *   p [L][E] f64 (> 0), C [M] f64, pi [M] f64 (the share of tokens whose
 *   trajectory reaches each server; a server with pi_m <= 0 gets no replica);
 *   placement [L][M][E] u8 in/out, used [M] f64 in/out (b_m),
 *   replicas [M] i32 out (replicas deployed per server).
 * Needs L * E <= 16384, L <= 1024, M <= 32. A group id >= E sets
 * ORDERMOE_DEV_BAD_INDEX, a p <= 0 or NaN ORDERMOE_DEV_BAD_VALUE (the entry is
 * skipped); both are read with ordermoe_device_error. */
int ordermoe_replicate(const int32_t* group, const double* importance, const double* p,
                       const double* C, const double* pi, int L, int E, int M,
                       uint8_t* placement, double* used, int32_t* replicas,
                       ordermoe_stream_t stream);

/* Local group coverage (Eq. 32) of a placement: cover[l][m][g] = 1 when server
 * m hosts an expert of group g in layer l (g < E; entries of groups a layer
 * does not have stay 0), covered[l] = the number of such (m, g) pairs. The
 * coverage ratio of Section VI-G is sum covered / (M * sum n_groups).
 *   group [L][E] i32, placement [L][M][E] u8; cover [L][M][E] u8 out
 *   (nullable), covered [L] i32 out (nullable). */
int ordermoe_coverage(const int32_t* group, const uint8_t* placement, int L, int E, int M,
                      uint8_t* cover, int32_t* covered, ordermoe_stream_t stream);

/* ------------------------------------------------------------------------
 * The whole offline plan of Alg. 1 in one call: similarity and counts
 * (Section III-B, Eqs. 3-5), thresholds, grouping and importance (Eqs. 6,
 * 24-28), mandatory placement (Eqs. 29-31), redundant deployment (Eqs. 32-35)
 * and coverage (Eq. 32). Every output equals, bit for bit, what
 * ordermoe_similarity_no_logits, ordermoe_place, ordermoe_replicate and
 * ordermoe_coverage write when called in that order with the same arguments.
 * For E in {8, 16, 32, 64} and L * E <= 4096 the layers go in blocks of 512 logit columns
 * (8 layers of 64 experts; the last block in two halves when there are
 * several, so that less grouping and placement is left after the last GEMM):
 * the caller's stream computes a block's logits,
 * Gram and similarities while a side stream of the library, ordered behind it
 * by events, groups and places the block before; the call joins the side
 * stream back into the caller's before replication, so work queued on the
 * caller's stream afterwards sees every output (CUDA graph capture included).
 * The side stream is the device's, shared by all calls: calls from several
 * host threads are enqueued one at a time, and their side-stream work runs in
 * that order. Otherwise the steps run one after the other on the caller's
 * stream.
 *   Arguments as in those four calls: W_r [L][E][d] bf16, X_cal [N][d] bf16;
 *   p [L][E] f64, C [M] f64, pi [M] f64; sim [L][E][E] f32, counts [L][E] i32,
 *   group [L][E] i32, n_groups [L] i32, theta [L] f32, importance [L][E] f64
 *   (not nullable here), placement [L][M][E] u8, used [M] f64, status [1] i32
 *   (ORDERMOE_OK or ORDERMOE_ERR_CAPACITY, as ordermoe_place), replicas [M] i32,
 *   cover [L][M][E] u8 (nullable), covered [L] i32 (nullable).
 *   workspace: ordermoe_plan_workspace_bytes(L, E, N) bytes, 256-byte aligned.
 * Needs the limits of the four calls together (L * E <= 16384, L <= 1024,
 * M <= 32, d a multiple of 64). */
size_t ordermoe_plan_workspace_bytes(int L, int E, int64_t N);
int ordermoe_plan(const uint16_t* W_r, const uint16_t* X_cal, int L, int E, int d, int64_t N,
                  int k_freq, int M, double theta_min, double theta_max, double theta_single,
                  double alpha_f, double alpha_r, double lambda1, double lambda2, const double* p,
                  const double* C, const double* pi, float* sim, int32_t* counts, int32_t* group,
                  int32_t* n_groups, float* theta, double* importance, uint8_t* placement,
                  double* used, int32_t* status, int32_t* replicas, uint8_t* cover,
                  int32_t* covered, void* workspace, size_t workspace_bytes,
                  ordermoe_stream_t stream);

/* ------------------------------------------------------------------------
 * Edge cost of L layers' selection records (Section III-D/E). Servers are the
 * logical placement map; the delays are the model's, not this GPU's. Token t
 * starts at home[t] (Eq. 36); at layer l, slot j executed on server m pays
 *   the transfer z / B[s][m] + tau[s][m] when m != s, s the token's location
 *   (Eqs. 13-14), and the compute c / F[m] (Eq. 15);
 * the location after the layer is the server of slot 0 (Eq. 44). A slot whose
 * executed expert differs from its target adds Q_l(target, executed), the
 * fp32 loss table of layer l's tables (Eq. 18), to the loss (Eqs. 19-20).
 *   target, chosen_expert [L][T][k] i32, chosen_server [L][T][k] u8, home [T] u8;
 *   tables: L layers' selection tables, tables_stride bytes apart (only Qtab
 *   is read); F [M] flop/s, B [M][M] bytes/s (row = source), tau [M][M] s,
 *   z bytes per transfer, c flop per expert execution (all f64, device);
 *   delay [T] f64 out (s, Eq. 17 with one token per user), loss [T] f64 out,
 *   moves [T] i32 out (transfers). fp64, one running sum per token in
 *   (layer, slot) order. An index out of range sets ORDERMOE_DEV_BAD_INDEX
 *   (detail: the token) and leaves that token's outputs unwritten. */
int ordermoe_trajectory_cost(const int32_t* target, const int32_t* chosen_expert,
                             const uint8_t* chosen_server, const uint8_t* home, int L, int T, int k,
                             int E, const void* tables, size_t tables_stride, int M,
                             const double* F, const double* B, const double* tau, double z,
                             double c, double* delay, double* loss, int32_t* moves,
                             ordermoe_stream_t stream);

/* Normalised utility (Eq. 23) and weight adaptation (Eq. 45) over T users of
 * one token each: T~ = delay / delay_ref (delay_ref: the same tokens under pure
 * exact execution on the same deployment), Q~ = loss / qmax;
 *   U = omega_T sum T~ + omega_Q sum Q~, Tbar = mean T~, Qbar = mean Q~,
 *   omega_Q' = clamp(omega_Q + kappa (Qbar - Tbar), 0, 1), omega_T' = 1 - omega_Q'.
 * out [5] f64 device: {U, Tbar, Qbar, omega_T', omega_Q'}. fp64 sums in a fixed
 * order (strided per thread, then a fixed tree). A delay_ref <= 0 sets
 * ORDERMOE_DEV_BAD_VALUE and the token is skipped. The caller rebuilds the
 * selection tables with the new weights (ordermoe_build_tables) once per
 * observation window. */
int ordermoe_utility(const double* delay, const double* delay_ref, const double* loss, int T,
                     double qmax, double omega_T, double omega_Q, double kappa, double* out,
                     ordermoe_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* ORDERMOE_H */
