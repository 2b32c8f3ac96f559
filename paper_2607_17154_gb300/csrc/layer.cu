// One MoE layer forward through the hot path: route_select -> dispatch ->
// expert gate/up -> expert down -> combine, with its scratch carved from one
// caller-provided buffer. With host_io the inputs are copied host -> device
// and the output device -> host on the same stream.
#include <mutex>

#include "common.cuh"

namespace om {
int dispatch_launch(const int32_t* chosen, const uint16_t* X, int T, int k, int E, int d,
                    int32_t* offsets, int32_t* row_token, int32_t* row_of, uint16_t* X_perm,
                    int32_t* hist, cudaStream_t stream);
size_t dispatch_workspace_bytes(int64_t n, int E);

struct LayerScratch {
  int32_t *topk_idx, *chosen, *offsets, *row_token, *row_of, *hist;
  float *topk_w, *qhat;
  uint8_t *server, *kind, *loc, *home;
  uint16_t *X_perm, *H, *Y_perm, *X, *y;
  size_t bytes;
};

static size_t up256(size_t v) { return (v + 255) & ~size_t(255); }

// Carves the scratch; with base == nullptr only computes its size.
static LayerScratch carve(uint8_t* base, int T, int E, int d, int dff, int k) {
  LayerScratch s{};
  size_t off = 0;
  const size_t R = (size_t)T * k;
  auto take = [&](size_t bytes) {
    uint8_t* p = base ? base + off : nullptr;
    off += up256(bytes);
    return p;
  };
  s.topk_idx = reinterpret_cast<int32_t*>(take(R * 4));
  s.topk_w = reinterpret_cast<float*>(take(R * 4));
  s.chosen = reinterpret_cast<int32_t*>(take(R * 4));
  s.server = take(R);
  s.kind = take(R);
  s.offsets = reinterpret_cast<int32_t*>(take((E + 1) * 4));
  s.row_token = reinterpret_cast<int32_t*>(take(R * 4));
  s.row_of = reinterpret_cast<int32_t*>(take(R * 4));
  s.hist = reinterpret_cast<int32_t*>(take(dispatch_workspace_bytes((int64_t)R, E)));
  s.X_perm = reinterpret_cast<uint16_t*>(take(R * d * 2));
  s.H = reinterpret_cast<uint16_t*>(take(R * dff * 2));
  s.Y_perm = reinterpret_cast<uint16_t*>(take(R * d * 2));
  s.loc = take(T);
  s.qhat = reinterpret_cast<float*>(take((size_t)T * 4));
  s.home = take(T);
  s.X = reinterpret_cast<uint16_t*>(take((size_t)T * d * 2));
  s.y = reinterpret_cast<uint16_t*>(take((size_t)T * d * 2));
  s.bytes = off;
  return s;
}

int gate_up_launch(const uint16_t* X_perm, const int32_t* offsets, int R, const uint16_t* W1,
                   const uint16_t* W3, int E, int d, int dff, uint16_t* H, cudaStream_t stream);
int down_launch(const uint16_t* H, const int32_t* offsets, int R, const uint16_t* W2, int E, int d,
                int dff, uint16_t* Y, cudaStream_t stream);

}  // namespace om

using namespace om;

extern "C" int ordermoe_route_select(const uint16_t* X, const uint16_t* W_r, const float* logits_in,
                                     int T, int E, int d, int k, int renorm, const void* tables,
                                     size_t tables_bytes_, const uint8_t* home, uint8_t* loc,
                                     float* qhat, float* logits_out, int32_t* topk_idx,
                                     float* topk_w, int32_t* chosen_expert,
                                     uint8_t* chosen_server, uint8_t* kind, int32_t* counters,
                                     ordermoe_stream_t stream);
extern "C" int ordermoe_route_select_lookahead(
    const uint16_t* X, const uint16_t* W_r, const float* logits_in, int T, int E, int d, int k,
    int renorm, const void* tables, size_t tables_stride, int H, const float* P,
    const uint8_t* home, uint8_t* loc, float* qhat, float* logits_out, int32_t* topk_idx,
    float* topk_w, int32_t* chosen_expert, uint8_t* chosen_server, uint8_t* kind,
    int32_t* counters, ordermoe_stream_t stream);
extern "C" int ordermoe_combine(const uint16_t* Y_perm, const int32_t* row_of,
                                const float* topk_w, int T, int k, int d, uint16_t* y,
                                ordermoe_stream_t stream);

// Second staging set (X, home, y) of the batched entry point.
static size_t batch_extra_bytes(int T_max, int d) {
  return up256((size_t)T_max * d * 2) * 2 + up256((size_t)T_max);
}

// Copy streams and events of the batched entry point, one set per device,
// shared by every call: a call holds `enq` while it enqueues, so calls from
// several host threads cannot interleave their event records.
struct BatchStreams {
  std::mutex enq;
  cudaStream_t h2d = nullptr, d2h = nullptr;
  cudaEvent_t start, end, in_ready[2], x_free[2], y_ready[2], y_free[2];
  bool ok = false;
};

static BatchStreams* batch_streams() {
  static std::mutex mu;
  static BatchStreams per_dev[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
  std::lock_guard<std::mutex> g(mu);
  BatchStreams& b = per_dev[dev];
  if (!b.ok) {
    const unsigned fl = cudaEventDisableTiming;
    bool good = cudaStreamCreateWithFlags(&b.h2d, cudaStreamNonBlocking) == cudaSuccess &&
                cudaStreamCreateWithFlags(&b.d2h, cudaStreamNonBlocking) == cudaSuccess &&
                cudaEventCreateWithFlags(&b.start, fl) == cudaSuccess &&
                cudaEventCreateWithFlags(&b.end, fl) == cudaSuccess;
    for (int i = 0; i < 2 && good; ++i)
      good = cudaEventCreateWithFlags(&b.in_ready[i], fl) == cudaSuccess &&
             cudaEventCreateWithFlags(&b.x_free[i], fl) == cudaSuccess &&
             cudaEventCreateWithFlags(&b.y_ready[i], fl) == cudaSuccess &&
             cudaEventCreateWithFlags(&b.y_free[i], fl) == cudaSuccess;
    if (!good) return nullptr;
    b.ok = true;
  }
  return &b;
}

extern "C" size_t ordermoe_layer_scratch_bytes(int T_max, int E, int d, int dff, int k) {
  if (T_max <= 0 || E <= 0 || E > ORDERMOE_MAX_EXPERTS || d <= 0 || dff <= 0 || k <= 0 ||
      k > ORDERMOE_MAX_TOPK)
    return 0;
  return carve(nullptr, T_max, E, d, dff, k).bytes;
}

// Checks of the layer descriptor shared by the single-call entry points.
static int check_layer(const ordermoe_layer_desc* L, int T, const char* who) {
  if (!L) return fail(ORDERMOE_ERR_INVALID_ARG, "%s: null layer", who);
  if (T < 0 || T > L->T_max) return fail(ORDERMOE_ERR_INVALID_ARG, "%s: need 0 <= T <= T_max", who);
  if (!L->W_r || !L->W1 || !L->W3 || !L->W2 || !L->tables || !L->scratch)
    return fail(ORDERMOE_ERR_INVALID_ARG, "%s: null pointer in the layer", who);
  if ((reinterpret_cast<uintptr_t>(L->scratch) & 255u) != 0)
    return fail(ORDERMOE_ERR_INVALID_ARG, "%s: scratch must be 256-byte aligned", who);
  const size_t need = ordermoe_layer_scratch_bytes(L->T_max, L->E, L->d, L->dff, L->k);
  if (need == 0 || L->scratch_bytes < need)
    return fail(ORDERMOE_ERR_INVALID_ARG, "%s: scratch too small or bad shape", who);
  if (L->d % 256 != 0 || L->dff % 128 != 0 || L->k > L->E)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "%s: need d %% 256 == 0, dff %% 128 == 0, k <= E", who);
  if (!aligned16(L->W_r) || !aligned16(L->W1) || !aligned16(L->W3) || !aligned16(L->W2))
    return fail(ORDERMOE_ERR_INVALID_ARG, "%s: weights must be 16-byte aligned", who);
  return ORDERMOE_OK;
}

extern "C" int ordermoe_combine_residual_norm(const uint16_t* Y_perm, const int32_t* row_of,
                                              const float* topk_w, const uint16_t* h, int T, int k,
                                              int d, float eps, uint16_t* h_out, uint16_t* x_out,
                                              ordermoe_stream_t stream);

extern "C" int ordermoe_layer_forward_residual(const ordermoe_layer_desc* L, int T,
                                               const uint16_t* x, const uint16_t* h,
                                               const uint8_t* home, uint8_t* loc, float* qhat,
                                               float eps, uint16_t* h_out, uint16_t* x_out,
                                               float* logits_out, int32_t* counters,
                                               ordermoe_stream_t stream) {
  OM_TRACE();
  int rc = check_layer(L, T, "layer_forward_residual");
  if (rc || T == 0) return rc;
  if (!x || !h || !home || !h_out || !x_out)
    return fail(ORDERMOE_ERR_INVALID_ARG, "layer_forward_residual: null x/h/home/h_out/x_out");
  if (!aligned16(x) || !aligned16(h) || !aligned16(h_out) || !aligned16(x_out))
    return fail(ORDERMOE_ERR_INVALID_ARG, "layer_forward_residual: x, h, h_out, x_out must be 16-byte aligned");
  if ((loc == nullptr) != (qhat == nullptr))
    return fail(ORDERMOE_ERR_INVALID_ARG, "layer_forward_residual: give both loc and qhat, or neither");
  const int E = L->E, d = L->d, dff = L->dff, k = L->k, R = T * k;
  LayerScratch s = carve(static_cast<uint8_t*>(L->scratch), L->T_max, E, d, dff, k);
  if (L->lookahead_H > 1)
    rc = ordermoe_route_select_lookahead(x, L->W_r, nullptr, T, E, d, k, L->renorm, L->tables,
                                         L->tables_stride, L->lookahead_H, L->P, home, loc, qhat,
                                         logits_out, s.topk_idx, s.topk_w, s.chosen, s.server,
                                         s.kind, counters, stream);
  else
    rc = ordermoe_route_select(x, L->W_r, nullptr, T, E, d, k, L->renorm, L->tables,
                               L->tables_bytes, home, loc, qhat, logits_out, s.topk_idx, s.topk_w,
                               s.chosen, s.server, s.kind, counters, stream);
  if (rc) return rc;
  rc = dispatch_launch(s.chosen, x, T, k, E, d, s.offsets, s.row_token, s.row_of, s.X_perm, s.hist,
                       stream);
  if (rc) return rc;
  rc = gate_up_launch(s.X_perm, s.offsets, R, L->W1, L->W3, E, d, dff, s.H, stream);
  if (rc) return rc;
  rc = down_launch(s.H, s.offsets, R, L->W2, E, d, dff, s.Y_perm, stream);
  if (rc) return rc;
  return ordermoe_combine_residual_norm(s.Y_perm, s.row_of, s.topk_w, h, T, k, d, eps, h_out,
                                        x_out, stream);
}

extern "C" int ordermoe_layer_forward(const ordermoe_layer_desc* L, int T, const uint16_t* X,
                                      const uint8_t* home, uint8_t* loc, float* qhat, uint16_t* y,
                                      int32_t* counters, int host_io, ordermoe_stream_t stream) {
  OM_TRACE();
  int rc0 = check_layer(L, T, "layer_forward");
  if (rc0) return rc0;
  if (T == 0) return ORDERMOE_OK;
  if (!X || !home || !y) return fail(ORDERMOE_ERR_INVALID_ARG, "layer_forward: null X/home/y");
  if ((loc == nullptr) != (qhat == nullptr))
    return fail(ORDERMOE_ERR_INVALID_ARG, "layer_forward: give both loc and qhat, or neither");
  const int E = L->E, d = L->d, dff = L->dff, k = L->k, R = T * k;
  LayerScratch s = carve(static_cast<uint8_t*>(L->scratch), L->T_max, E, d, dff, k);
  cudaStream_t st = stream;
  const uint16_t* Xd = X;
  const uint8_t* homed = home;
  uint8_t* locd = loc;
  float* qd = qhat;
  uint16_t* yd = y;
  if (!host_io && (!aligned16(X) || !aligned16(y)))
    return fail(ORDERMOE_ERR_INVALID_ARG, "layer_forward: X and y must be 16-byte aligned");
  if (host_io) {
    OM_CUDA(cudaMemcpyAsync(s.X, X, (size_t)T * d * 2, cudaMemcpyHostToDevice, st));
    OM_CUDA(cudaMemcpyAsync(s.home, home, (size_t)T, cudaMemcpyHostToDevice, st));
    Xd = s.X;
    homed = s.home;
    yd = s.y;
    if (loc) {
      OM_CUDA(cudaMemcpyAsync(s.loc, loc, (size_t)T, cudaMemcpyHostToDevice, st));
      OM_CUDA(cudaMemcpyAsync(s.qhat, qhat, (size_t)T * 4, cudaMemcpyHostToDevice, st));
      locd = s.loc;
      qd = s.qhat;
    }
  }
  int rc;
  if (L->lookahead_H > 1)
    rc = ordermoe_route_select_lookahead(Xd, L->W_r, nullptr, T, E, d, k, L->renorm, L->tables,
                                         L->tables_stride, L->lookahead_H, L->P, homed, locd, qd,
                                         nullptr, s.topk_idx, s.topk_w, s.chosen, s.server, s.kind,
                                         counters, stream);
  else
    rc = ordermoe_route_select(Xd, L->W_r, nullptr, T, E, d, k, L->renorm, L->tables,
                               L->tables_bytes, homed, locd, qd, nullptr, s.topk_idx, s.topk_w,
                               s.chosen, s.server, s.kind, counters, stream);
  if (rc) return rc;
  rc = dispatch_launch(s.chosen, Xd, T, k, E, d, s.offsets, s.row_token, s.row_of, s.X_perm,
                       s.hist, st);
  if (rc) return rc;
  rc = gate_up_launch(s.X_perm, s.offsets, R, L->W1, L->W3, E, d, dff, s.H, st);
  if (rc) return rc;
  rc = down_launch(s.H, s.offsets, R, L->W2, E, d, dff, s.Y_perm, st);
  if (rc) return rc;
  rc = ordermoe_combine(s.Y_perm, s.row_of, s.topk_w, T, k, d, yd, stream);
  if (rc) return rc;
  if (host_io) {
    OM_CUDA(cudaMemcpyAsync(y, s.y, (size_t)T * d * 2, cudaMemcpyDeviceToHost, st));
    if (loc) {
      OM_CUDA(cudaMemcpyAsync(loc, s.loc, (size_t)T, cudaMemcpyDeviceToHost, st));
      OM_CUDA(cudaMemcpyAsync(qhat, s.qhat, (size_t)T * 4, cudaMemcpyDeviceToHost, st));
    }
  }
  return ORDERMOE_OK;
}

extern "C" size_t ordermoe_layer_batches_scratch_bytes(int T_max, int E, int d, int dff, int k) {
  const size_t base = ordermoe_layer_scratch_bytes(T_max, E, d, dff, k);
  return base ? base + batch_extra_bytes(T_max, d) : 0;
}

extern "C" int ordermoe_layer_forward_batches(const ordermoe_layer_desc* L, int nbatch, int T,
                                              const uint16_t* X, const uint8_t* home, uint16_t* y,
                                              int32_t* counters, ordermoe_stream_t stream) {
  OM_TRACE();
  if (!L) return fail(ORDERMOE_ERR_INVALID_ARG, "layer_forward_batches: null layer");
  if (nbatch < 0 || T < 0 || T > L->T_max)
    return fail(ORDERMOE_ERR_INVALID_ARG, "layer_forward_batches: need nbatch >= 0, 0 <= T <= T_max");
  if (!L->W_r || !L->W1 || !L->W3 || !L->W2 || !L->tables || !L->scratch)
    return fail(ORDERMOE_ERR_INVALID_ARG, "layer_forward_batches: null pointer in the layer");
  if ((reinterpret_cast<uintptr_t>(L->scratch) & 255u) != 0)
    return fail(ORDERMOE_ERR_INVALID_ARG, "layer_forward_batches: scratch must be 256-byte aligned");
  const size_t need = ordermoe_layer_batches_scratch_bytes(L->T_max, L->E, L->d, L->dff, L->k);
  if (need == 0 || L->scratch_bytes < need)
    return fail(ORDERMOE_ERR_INVALID_ARG, "layer_forward_batches: scratch too small or bad shape");
  if (L->d % 256 != 0 || L->dff % 128 != 0 || L->k > L->E)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "layer_forward_batches: need d %% 256 == 0, dff %% 128 == 0, k <= E");
  if (!aligned16(L->W_r) || !aligned16(L->W1) || !aligned16(L->W3) || !aligned16(L->W2))
    return fail(ORDERMOE_ERR_INVALID_ARG, "layer_forward_batches: weights must be 16-byte aligned");
  if (T == 0 || nbatch == 0) return ORDERMOE_OK;
  if (!X || !home || !y) return fail(ORDERMOE_ERR_INVALID_ARG, "layer_forward_batches: null X/home/y");
  BatchStreams* bs = batch_streams();
  if (!bs) return fail(ORDERMOE_ERR_CUDA, "layer_forward_batches: could not create its copy streams");
  const int E = L->E, d = L->d, dff = L->dff, k = L->k, R = T * k;
  LayerScratch s = carve(static_cast<uint8_t*>(L->scratch), L->T_max, E, d, dff, k);
  // staging slot 0 is the layer scratch's X / home / y, slot 1 follows the layer scratch
  uint8_t* extra = static_cast<uint8_t*>(L->scratch) + s.bytes;
  uint16_t* Xs[2] = {s.X, reinterpret_cast<uint16_t*>(extra)};
  uint16_t* ys[2] = {s.y, reinterpret_cast<uint16_t*>(extra + up256((size_t)L->T_max * d * 2))};
  uint8_t* hs[2] = {s.home, extra + 2 * up256((size_t)L->T_max * d * 2)};
  cudaStream_t st = stream;
  const size_t xb = (size_t)T * d * 2;
  std::lock_guard<std::mutex> hold(bs->enq);
  // the copy streams start after everything already on the caller's stream
  OM_CUDA(cudaEventRecord(bs->start, st));
  OM_CUDA(cudaStreamWaitEvent(bs->h2d, bs->start, 0));
  OM_CUDA(cudaStreamWaitEvent(bs->d2h, bs->start, 0));
  auto ck = [](cudaError_t e, const char* what) { return e == cudaSuccess ? 0 : cuda_fail(e, what); };
  int rc = 0;
  for (int b = 0; b < nbatch && !rc; ++b) {
    const int sl = b & 1;
    // batch b's inputs: after batch b - 2 has finished reading this slot
    if (b >= 2 && (rc = ck(cudaStreamWaitEvent(bs->h2d, bs->x_free[sl], 0), "wait x_free"))) break;
    if ((rc = ck(cudaMemcpyAsync(Xs[sl], X + (size_t)b * T * d, xb, cudaMemcpyHostToDevice, bs->h2d),
                 "copy X")))
      break;
    if ((rc = ck(cudaMemcpyAsync(hs[sl], home + (size_t)b * T, (size_t)T, cudaMemcpyHostToDevice,
                                 bs->h2d), "copy home")))
      break;
    if ((rc = ck(cudaEventRecord(bs->in_ready[sl], bs->h2d), "record in_ready"))) break;
    if ((rc = ck(cudaStreamWaitEvent(st, bs->in_ready[sl], 0), "wait in_ready"))) break;
    if (L->lookahead_H > 1)
      rc = ordermoe_route_select_lookahead(Xs[sl], L->W_r, nullptr, T, E, d, k, L->renorm, L->tables,
                                           L->tables_stride, L->lookahead_H, L->P, hs[sl], nullptr,
                                           nullptr, nullptr, s.topk_idx, s.topk_w, s.chosen,
                                           s.server, s.kind, counters, st);
    else
      rc = ordermoe_route_select(Xs[sl], L->W_r, nullptr, T, E, d, k, L->renorm, L->tables,
                                 L->tables_bytes, hs[sl], nullptr, nullptr, nullptr, s.topk_idx,
                                 s.topk_w, s.chosen, s.server, s.kind, counters, st);
    if (rc) break;
    rc = dispatch_launch(s.chosen, Xs[sl], T, k, E, d, s.offsets, s.row_token, s.row_of, s.X_perm,
                         s.hist, st);
    if (rc) break;
    if ((rc = ck(cudaEventRecord(bs->x_free[sl], st), "record x_free"))) break;  // slot's X, home read
    rc = gate_up_launch(s.X_perm, s.offsets, R, L->W1, L->W3, E, d, dff, s.H, st);
    if (rc) break;
    rc = down_launch(s.H, s.offsets, R, L->W2, E, d, dff, s.Y_perm, st);
    if (rc) break;
    // the output slot: after batch b - 2's copy out has read it
    if (b >= 2 && (rc = ck(cudaStreamWaitEvent(st, bs->y_free[sl], 0), "wait y_free"))) break;
    rc = ordermoe_combine(s.Y_perm, s.row_of, s.topk_w, T, k, d, ys[sl], st);
    if (rc) break;
    if ((rc = ck(cudaEventRecord(bs->y_ready[sl], st), "record y_ready"))) break;
    if ((rc = ck(cudaStreamWaitEvent(bs->d2h, bs->y_ready[sl], 0), "wait y_ready"))) break;
    if ((rc = ck(cudaMemcpyAsync(y + (size_t)b * T * d, ys[sl], xb, cudaMemcpyDeviceToHost, bs->d2h),
                 "copy y")))
      break;
    if ((rc = ck(cudaEventRecord(bs->y_free[sl], bs->d2h), "record y_free"))) break;
  }
  // the caller's stream is ordered after every copy of this call, on every
  // exit once the copy streams have been forked (the error of a failed step
  // stays the one returned)
  cudaError_t e = cudaEventRecord(bs->end, bs->h2d);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(st, bs->end, 0);
  if (e == cudaSuccess) e = cudaEventRecord(bs->end, bs->d2h);
  if (e == cudaSuccess) e = cudaStreamWaitEvent(st, bs->end, 0);
  if (!rc && e != cudaSuccess) rc = cuda_fail(e, "layer_forward_batches: join");
  return rc;
}
