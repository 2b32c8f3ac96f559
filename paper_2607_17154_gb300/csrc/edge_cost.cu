// Edge cost of the selection records (Section III-D/E) and the runtime weight
// adaptation (Section V-D):
//   ordermoe_trajectory_cost: per-token delay (Eqs. 13-17), substitution loss
//     (Eqs. 18-20) and transfer count of L layers' decisions;
//   ordermoe_utility: normalised utility (Eq. 23) and the update of
//     omega_T / omega_Q (Eq. 45).
#include "common.cuh"

namespace om {

static __device__ unsigned long long g_err_cost = 0;

int read_clear_err_cost(unsigned long long* out) {
  unsigned long long zero = 0;
  OM_CUDA(cudaMemcpyFromSymbol(out, g_err_cost, sizeof(*out)));
  OM_CUDA(cudaMemcpyToSymbol(g_err_cost, &zero, sizeof(zero)));
  return ORDERMOE_OK;
}

constexpr size_t kQtabOffset = 832;  // Qtab [E][E] f32 in a layer's tables (ordermoe.h)

// One thread per token: the layers and slots in order, one fp64 running sum
// each for delay and loss. The location starts at home (Eq. 36) and moves to
// the server of slot 0 after every layer (Eq. 44); each slot pays the
// transfer from the location when it runs elsewhere (Eqs. 13-14) and the
// compute on its server (Eq. 15).
__global__ void __launch_bounds__(128) trajectory_cost_kernel(
    const int32_t* __restrict__ target, const int32_t* __restrict__ chosen,
    const uint8_t* __restrict__ server, const uint8_t* __restrict__ home, int L, int T, int k,
    int E, const uint8_t* __restrict__ tables, size_t stride, int M, const double* __restrict__ F,
    const double* __restrict__ B, const double* __restrict__ tau, double z, double c,
    double* __restrict__ delay, double* __restrict__ loss, int32_t* __restrict__ moves) {
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= T) return;
  int s = home[t];
  if (s >= M) {
    report(&g_err_cost, ORDERMOE_DEV_BAD_INDEX, t);
    return;
  }
  double d = 0.0, q = 0.0;
  int n = 0;
  for (int l = 0; l < L; ++l) {
    const float* Qtab = reinterpret_cast<const float*>(tables + (size_t)l * stride + kQtabOffset);
    int next = s;
    for (int j = 0; j < k; ++j) {
      const size_t i = ((size_t)l * T + t) * k + j;
      const int r = target[i], kk = chosen[i], m = server[i];
      if (r < 0 || r >= E || kk < 0 || kk >= E || m >= M) {
        report(&g_err_cost, ORDERMOE_DEV_BAD_INDEX, t);
        return;
      }
      double trans = 0.0;
      if (m != s) {
        trans = __dadd_rn(__ddiv_rn(z, B[s * M + m]), tau[s * M + m]);
        ++n;
      }
      const double comp = __ddiv_rn(c, F[m]);
      d = __dadd_rn(d, __dadd_rn(trans, comp));
      if (kk != r) q = __dadd_rn(q, static_cast<double>(Qtab[r * E + kk]));
      if (j == 0) next = m;
    }
    s = next;
  }
  delay[t] = d;
  loss[t] = q;
  moves[t] = n;
}

constexpr int kUtilThreads = 1024;

// One block: fp64 partial sums of T~ = delay / delay_ref and Q~ = loss / qmax
// (strided over the tokens, then a fixed tree), Eq. 23, then Eq. 45.
__global__ void __launch_bounds__(kUtilThreads) utility_kernel(
    const double* __restrict__ delay, const double* __restrict__ delay_ref,
    const double* __restrict__ loss, int T, double qmax, double omega_T, double omega_Q,
    double kappa, double* __restrict__ out) {
  __shared__ double st[kUtilThreads / 32], sq[kUtilThreads / 32];
  double a = 0.0, b = 0.0;
  for (int t = threadIdx.x; t < T; t += blockDim.x) {
    const double r = delay_ref[t];
    if (!(r > 0.0)) {
      report(&g_err_cost, ORDERMOE_DEV_BAD_VALUE, t);
      continue;
    }
    a = __dadd_rn(a, __ddiv_rn(delay[t], r));
    b = __dadd_rn(b, __ddiv_rn(loss[t], qmax));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    a = __dadd_rn(a, __shfl_xor_sync(0xffffffffu, a, o));
    b = __dadd_rn(b, __shfl_xor_sync(0xffffffffu, b, o));
  }
  const int w = threadIdx.x >> 5;
  if ((threadIdx.x & 31) == 0) {
    st[w] = a;
    sq[w] = b;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double sa = 0.0, sb = 0.0;
    for (int i = 0; i < (int)(blockDim.x >> 5); ++i) {
      sa = __dadd_rn(sa, st[i]);
      sb = __dadd_rn(sb, sq[i]);
    }
    const double tbar = __ddiv_rn(sa, static_cast<double>(T));
    const double qbar = __ddiv_rn(sb, static_cast<double>(T));
    double wq = __dadd_rn(omega_Q, __dmul_rn(kappa, __dsub_rn(qbar, tbar)));
    wq = fmin(1.0, fmax(0.0, wq));
    out[0] = __dadd_rn(__dmul_rn(omega_T, sa), __dmul_rn(omega_Q, sb));
    out[1] = tbar;
    out[2] = qbar;
    out[3] = __dsub_rn(1.0, wq);
    out[4] = wq;
  }
}

}  // namespace om

using namespace om;

extern "C" int ordermoe_trajectory_cost(const int32_t* target, const int32_t* chosen_expert,
                                        const uint8_t* chosen_server, const uint8_t* home, int L,
                                        int T, int k, int E, const void* tables,
                                        size_t tables_stride, int M, const double* F,
                                        const double* B, const double* tau, double z, double c,
                                        double* delay, double* loss, int32_t* moves,
                                        ordermoe_stream_t stream) {
  OM_TRACE();
  if (L <= 0 || T < 0 || k <= 0 || k > ORDERMOE_MAX_TOPK || E <= 0 || E > ORDERMOE_MAX_EXPERTS ||
      M <= 0 || M > ORDERMOE_MAX_SERVERS)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE,
                "trajectory_cost: need L >= 1, T >= 0, 1 <= k <= 8, 1 <= E <= 64, 1 <= M <= 32");
  if (T == 0) return ORDERMOE_OK;
  if (!target || !chosen_expert || !chosen_server || !home || !tables || !F || !B || !tau ||
      !delay || !loss || !moves)
    return fail(ORDERMOE_ERR_INVALID_ARG, "trajectory_cost: null pointer");
  if (L > 1 && tables_stride < ordermoe_tables_bytes(E, M))
    return fail(ORDERMOE_ERR_INVALID_ARG, "trajectory_cost: tables_stride below one layer's tables");
  trajectory_cost_kernel<<<(T + 127) / 128, 128, 0, stream>>>(
      target, chosen_expert, chosen_server, home, L, T, k, E, static_cast<const uint8_t*>(tables),
      tables_stride, M, F, B, tau, z, c, delay, loss, moves);
  OM_LAUNCHED("trajectory_cost_kernel");
  return ORDERMOE_OK;
}

extern "C" int ordermoe_utility(const double* delay, const double* delay_ref, const double* loss,
                                int T, double qmax, double omega_T, double omega_Q, double kappa,
                                double* out, ordermoe_stream_t stream) {
  OM_TRACE();
  if (T <= 0) return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "utility: need T >= 1");
  if (!(qmax > 0.0)) return fail(ORDERMOE_ERR_INVALID_ARG, "utility: need qmax > 0");
  if (!delay || !delay_ref || !loss || !out) return fail(ORDERMOE_ERR_INVALID_ARG, "utility: null pointer");
  utility_kernel<<<1, kUtilThreads, 0, stream>>>(delay, delay_ref, loss, T, qmax, omega_T, omega_Q,
                                                 kappa, out);
  OM_LAUNCHED("utility_kernel");
  return ORDERMOE_OK;
}
