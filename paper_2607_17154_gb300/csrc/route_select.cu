// Router + softmax + top-k + server-expert selection (Alg. 2, H = 1), and the
// per-layer selection tables it reads (Eqs. 7, 18, 37, 38).
#include <cstring>

#include "common.cuh"

namespace om {

static __device__ unsigned long long g_err_route = 0;

int read_clear_err_route(unsigned long long* out) {
  unsigned long long zero = 0;
  OM_CUDA(cudaMemcpyFromSymbol(out, g_err_route, sizeof(*out)));
  OM_CUDA(cudaMemcpyToSymbol(g_err_route, &zero, sizeof(zero)));
  return ORDERMOE_OK;
}

// Byte layout of the tables buffer (documented in ordermoe.h).
constexpr int kTabMagic = 0x4f4d5442;
constexpr size_t kOffPmask = 64, kOffSubst = 320, kOffQtab = 832;
__host__ __device__ inline size_t off_cq(int E) { return kOffQtab + sizeof(float) * E * E; }
__host__ __device__ inline size_t off_a(int E) { return off_cq(E) + sizeof(float) * E * E; }
__host__ __device__ inline size_t tables_bytes(int E, int M) {
  size_t b = off_a(E) + sizeof(float) * (size_t)M * M * M;
  return (b + 255) & ~size_t(255);
}

// ---------------------------------------------------------------------------
// Tables. One block; fp64 terms use explicit round-to-nearest operations so
// that no multiply-add is fused.
__global__ void build_tables_kernel(const float* __restrict__ sim, const int32_t* __restrict__ group,
                                    const uint8_t* __restrict__ placement, int E, int M,
                                    float theta, float qbar, const double* __restrict__ F,
                                    const double* __restrict__ B, const double* __restrict__ tau,
                                    double z, double c, double omega_T, double omega_Q,
                                    uint8_t* __restrict__ tab) {
  int32_t* hdr = reinterpret_cast<int32_t*>(tab);
  float* hdrf = reinterpret_cast<float*>(tab);
  uint32_t* pmask = reinterpret_cast<uint32_t*>(tab + kOffPmask);
  unsigned long long* subst = reinterpret_cast<unsigned long long*>(tab + kOffSubst);
  float* Qtab = reinterpret_cast<float*>(tab + kOffQtab);
  float* Cq = reinterpret_cast<float*>(tab + off_cq(E));
  float* A = reinterpret_cast<float*>(tab + off_a(E));
  const int tid = threadIdx.x;
  if (tid == 0) {
    hdr[0] = kTabMagic; hdr[1] = E; hdr[2] = M; hdr[3] = 0;
    hdrf[4] = theta; hdrf[5] = qbar;
  }
  for (int e = tid; e < 64; e += blockDim.x) {
    uint32_t pm = 0;
    unsigned long long sb = 0;
    if (e < E) {
      for (int m = 0; m < M; ++m)
        if (placement[m * E + e]) pm |= 1u << m;
      for (int k = 0; k < E; ++k) {
        const float s = sim[e * E + k];
        if (k != e && group[k] == group[e] && s >= theta) sb |= 1ull << k;
      }
    }
    pmask[e] = pm;
    subst[e] = sb;
  }
  for (int i = tid; i < E * E; i += blockDim.x) {
    const int r = i / E, k = i % E;
    const float s = sim[i];
    float q = 0.0f;
    if (k != r) q = __fmul_rn(0.5f, __fsub_rn(1.0f, (1.0f < s) ? 1.0f : s));  // Eq. 18
    Qtab[i] = q;
    float cq = 0.0f;
    if (q != 0.0f)
      cq = __double2float_rn(__ddiv_rn(__dmul_rn(omega_Q, static_cast<double>(q)),
                                       static_cast<double>(qbar)));
    Cq[i] = cq;
  }
  for (int i = tid; i < M * M * M; i += blockDim.x) {
    const int a = i / (M * M), s = (i / M) % M, m = i % M;
    const double dref = __ddiv_rn(c, F[a]);
    const double comp = __ddiv_rn(c, F[m]);
    double dl = comp;
    if (s != m) {
      const double trans = __dadd_rn(__ddiv_rn(z, B[s * M + m]), tau[s * M + m]);  // Eq. 37
      dl = __dadd_rn(trans, comp);
    }
    A[i] = __double2float_rn(__ddiv_rn(__dmul_rn(omega_T, dl), dref));  // Eq. 38, delay term
  }
}

// ---------------------------------------------------------------------------
// Router + top-k + selection. One warp per token.
//
// Router: lane l accumulates the fp32 partial dot products of 8-element
// chunks c = 8 l, 8 l + 256, ...; a butterfly reduction gives every lane all E
// logits. Top-k and softmax are then computed redundantly by every lane (E
// is at most 64), so the per-slot selection needs no further communication.
//
// Selection, per slot j in rank order (Eqs. 36-44): the candidates are the
// pairs (m, k') with k' = r (exact) or k' in R_{l,r} (Eq. 7), x_{m,k'} = 1,
// and for substitutes k' not yet used by the token and Qhat + Q(r,k') <= Qbar
// (Eq. 40). Lanes take candidates c = lane, lane + 32, ...; the cost of Eq. 38
// is A[a][s][m] + Cq[r][k'] (one fp32 add), packed with the tie-break fields
// into a 64-bit key whose warp-wide minimum is the argmin of Eq. 43. Costs
// are never negative, so the fp32 bit pattern orders them.
template <int EMAX>
__global__ void __launch_bounds__(256) route_select_kernel(
    const uint16_t* __restrict__ X, const uint16_t* __restrict__ Wr,
    const float* __restrict__ logits_in, int T, int E, int d, int k, int renorm,
    const uint8_t* __restrict__ tab, const uint8_t* __restrict__ home, uint8_t* __restrict__ loc,
    float* __restrict__ qhat, float* __restrict__ logits_out, int32_t* __restrict__ topk_idx,
    float* __restrict__ topk_w, int32_t* __restrict__ chosen_expert,
    uint8_t* __restrict__ chosen_server, uint8_t* __restrict__ kind_out,
    int32_t* __restrict__ counters, int stage_w) {
  __shared__ uint32_t s_pmask[64];
  __shared__ unsigned long long s_subst[64];
  __shared__ uint8_t s_sublist[64 * 64];
  __shared__ int s_nsub[64];
  __shared__ int s_kind[4];
  extern __shared__ __align__(16) float s_dyn[];  // Qtab[E*E], Cq[E*E], then W_r if staged
  float* s_Q = s_dyn;
  float* s_Cq = s_dyn + E * E;
  // W_r staged in shared memory when it fits (stage_w): every token of the
  // block then reads it at shared-memory latency instead of from L2.
  uint4* s_W = reinterpret_cast<uint4*>(s_dyn + ((2 * E * E + 3) & ~3));

  const int M = reinterpret_cast<const int32_t*>(tab)[2];
  if (reinterpret_cast<const int32_t*>(tab)[1] != E || M <= 0 || M > 32) {
    if (blockIdx.x == 0 && threadIdx.x == 0) report(&g_err_route, ORDERMOE_DEV_BAD_INDEX, -1);
    return;
  }
  const float qbar = reinterpret_cast<const float*>(tab)[5];
  const float* gQ = reinterpret_cast<const float*>(tab + kOffQtab);
  const float* gCq = reinterpret_cast<const float*>(tab + off_cq(E));
  const float* gA = reinterpret_cast<const float*>(tab + off_a(E));

  for (int i = threadIdx.x; i < 64; i += blockDim.x) {
    s_pmask[i] = reinterpret_cast<const uint32_t*>(tab + kOffPmask)[i];
    unsigned long long sb = reinterpret_cast<const unsigned long long*>(tab + kOffSubst)[i];
    s_subst[i] = sb;
    int n = 0;
    while (sb) {
      const int b = __ffsll(static_cast<long long>(sb)) - 1;
      s_sublist[i * 64 + n++] = static_cast<uint8_t>(b);
      sb &= sb - 1;
    }
    s_nsub[i] = n;
  }
  for (int i = threadIdx.x; i < E * E; i += blockDim.x) {
    s_Q[i] = gQ[i];
    s_Cq[i] = gCq[i];
  }
  if (stage_w && logits_in == nullptr) {
    const uint4* gw = reinterpret_cast<const uint4*>(Wr);
    for (int i = threadIdx.x; i < E * (d >> 3); i += blockDim.x) s_W[i] = __ldg(gw + i);
  }
  if (threadIdx.x < 4) s_kind[threadIdx.x] = 0;
  __syncthreads();

  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5;
  const int warps_total = gridDim.x * (blockDim.x >> 5);
  int kind_count[4] = {0, 0, 0, 0};

  for (int t = blockIdx.x * (blockDim.x >> 5) + warp; t < T; t += warps_total) {
    float lg[EMAX];
    if (logits_in != nullptr) {
#pragma unroll
      for (int e = 0; e < EMAX; ++e) lg[e] = (e < E) ? logits_in[(size_t)t * E + e] : 0.0f;
    } else {
#pragma unroll
      for (int e = 0; e < EMAX; ++e) lg[e] = 0.0f;
      const uint4* xr = reinterpret_cast<const uint4*>(X + (size_t)t * d);
      const int nvec = d >> 3;
      // X is streamed once from HBM: keep kBatch independent 16-byte loads
      // per lane in flight before using them; W_r stays in L1.
      constexpr int kBatch = 4;
      for (int c0 = lane; c0 < nvec; c0 += 32 * kBatch) {
        uint4 xv[kBatch];
#pragma unroll
        for (int b = 0; b < kBatch; ++b) {
          const int c = c0 + 32 * b;
          xv[b] = (c < nvec) ? __ldg(xr + c) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int b = 0; b < kBatch; ++b) {
          const int c = c0 + 32 * b;
          if (c >= nvec) break;
          const float x0 = bf16_lo(xv[b].x), x1 = bf16_hi(xv[b].x), x2 = bf16_lo(xv[b].y);
          const float x3 = bf16_hi(xv[b].y), x4 = bf16_lo(xv[b].z), x5 = bf16_hi(xv[b].z);
          const float x6 = bf16_lo(xv[b].w), x7 = bf16_hi(xv[b].w);
#pragma unroll
          for (int e = 0; e < EMAX; ++e) {
            if (e < E) {
              const uint4 wv = stage_w ? s_W[e * nvec + c]
                                       : __ldg(reinterpret_cast<const uint4*>(Wr + (size_t)e * d) + c);
              float a = lg[e];
              a = fmaf(x0, bf16_lo(wv.x), a); a = fmaf(x1, bf16_hi(wv.x), a);
              a = fmaf(x2, bf16_lo(wv.y), a); a = fmaf(x3, bf16_hi(wv.y), a);
              a = fmaf(x4, bf16_lo(wv.z), a); a = fmaf(x5, bf16_hi(wv.z), a);
              a = fmaf(x6, bf16_lo(wv.w), a); a = fmaf(x7, bf16_hi(wv.w), a);
              lg[e] = a;
            }
          }
        }
      }
#pragma unroll
      for (int e = 0; e < EMAX; ++e) {
        float v = lg[e];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        lg[e] = v;
      }
    }
    // logits out: lane e (and e + 32) writes expert e
    if (logits_out != nullptr) {
#pragma unroll
      for (int e = 0; e < EMAX; ++e)
        if (e < E && (e & 31) == lane) logits_out[(size_t)t * E + e] = lg[e];
    }
    bool bad = false;
#pragma unroll
    for (int e = 0; e < EMAX; ++e)
      if (e < E && isnan(lg[e])) bad = true;
    if (bad) {
      if (lane == 0) report(&g_err_route, ORDERMOE_DEV_NAN_LOGIT, t);
      continue;
    }
    // top-k by (logit desc, index asc)
    int idx[ORDERMOE_MAX_TOPK];
    unsigned long long used_targets = 0;
    for (int j = 0; j < k; ++j) {
      int best = -1;
      float bv = 0.0f;
#pragma unroll
      for (int e = 0; e < EMAX; ++e) {
        if (e < E && !((used_targets >> e) & 1ull)) {
          if (best < 0 || lg[e] > bv) { best = e; bv = lg[e]; }
        }
      }
      idx[j] = best;
      used_targets |= 1ull << best;
    }
    // softmax over all E in fp32, gate weights of the k slots
    float lmax = -INFINITY;
#pragma unroll
    for (int e = 0; e < EMAX; ++e)
      if (e < E) lmax = fmaxf(lmax, lg[e]);
    float denom = 0.0f;
#pragma unroll
    for (int e = 0; e < EMAX; ++e)
      if (e < E) denom += expf(lg[e] - lmax);
    float wsel[ORDERMOE_MAX_TOPK];
    float ssel = 0.0f;
    for (int j = 0; j < k; ++j) {
      float v = 0.0f;
#pragma unroll
      for (int e = 0; e < EMAX; ++e)
        if (e == idx[j]) v = lg[e];
      wsel[j] = expf(v - lmax) / denom;
      ssel += wsel[j];
    }
    if (lane == 0) {
      for (int j = 0; j < k; ++j) {
        topk_idx[(size_t)t * k + j] = idx[j];
        topk_w[(size_t)t * k + j] = renorm ? wsel[j] / ssel : wsel[j];
      }
    }

    // selection
    const int a = home[t];
    const int s = (loc != nullptr) ? loc[t] : a;  // no state given: first layer (Eq. 36)
    if (a >= M || s >= M) {
      if (lane == 0) report(&g_err_route, ORDERMOE_DEV_BAD_INDEX, t);
      continue;
    }
    const float* Aas = gA + ((size_t)a * M + s) * M;
    float q = (qhat != nullptr) ? qhat[t] : 0.0f;
    unsigned long long taken = used_targets;
    int first_server = s;
    for (int j = 0; j < k; ++j) {
      const int r = idx[j];
      const int nsub = s_nsub[r];
      const int ncand = (1 + nsub) * M;
      unsigned long long best = ~0ull;
      for (int cidx = lane; cidx < ncand; cidx += 32) {
        const int ki = cidx / M;
        const int m = cidx - ki * M;
        const int kk = (ki == 0) ? r : s_sublist[r * 64 + ki - 1];
        if (!((s_pmask[kk] >> m) & 1u)) continue;
        const bool sub = (ki != 0);
        float cost = __ldg(Aas + m);
        if (sub) {
          if ((taken >> kk) & 1ull) continue;
          if (!(__fadd_rn(q, s_Q[r * E + kk]) <= qbar)) continue;
          cost = __fadd_rn(cost, s_Cq[r * E + kk]);
        } else {
          cost = __fadd_rn(cost, 0.0f);
        }
        const unsigned long long key =
            (static_cast<unsigned long long>(__float_as_uint(cost)) << 32) |
            (static_cast<unsigned long long>(sub ? 1u : 0u) << 31) |
            (static_cast<unsigned long long>(m != s ? 1u : 0u) << 30) |
            (static_cast<unsigned long long>(m) << 8) | static_cast<unsigned long long>(kk);
        best = key < best ? key : best;
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long other = __shfl_xor_sync(0xffffffffu, best, o);
        best = other < best ? other : best;
      }
      int kstar, mstar, kd;
      if (best == ~0ull) {
        if (lane == 0) report(&g_err_route, ORDERMOE_DEV_NO_CANDIDATE, t);
        kstar = r; mstar = s; kd = 0;
      } else {
        kstar = static_cast<int>(best & 0xFFu);
        mstar = static_cast<int>((best >> 8) & 0xFFu);
        const int sub = static_cast<int>((best >> 31) & 1u);
        const int away = static_cast<int>((best >> 30) & 1u);
        kd = 2 * away + sub;
        if (sub) {
          taken |= 1ull << kstar;
          q = __fadd_rn(q, s_Q[r * E + kstar]);
        }
      }
      if (j == 0) first_server = mstar;
      if (lane == 0) {
        chosen_expert[(size_t)t * k + j] = kstar;
        chosen_server[(size_t)t * k + j] = static_cast<uint8_t>(mstar);
        kind_out[(size_t)t * k + j] = static_cast<uint8_t>(kd);
      }
      kind_count[kd]++;
    }
    if (lane == 0 && loc != nullptr) {
      loc[t] = static_cast<uint8_t>(first_server);
      qhat[t] = q;
    }
  }
  if (counters != nullptr) {
    if (lane == 0)
      for (int i = 0; i < 4; ++i)
        if (kind_count[i]) atomicAdd(&s_kind[i], kind_count[i]);
    __syncthreads();
    if (threadIdx.x < 4 && s_kind[threadIdx.x]) atomicAdd(&counters[threadIdx.x], s_kind[threadIdx.x]);
  }
}

}  // namespace om

using namespace om;

extern "C" size_t ordermoe_tables_bytes(int E, int M) {
  if (E <= 0 || E > ORDERMOE_MAX_EXPERTS || M <= 0 || M > ORDERMOE_MAX_SERVERS) return 0;
  return om::tables_bytes(E, M);
}

extern "C" int ordermoe_build_tables(const float* sim, const int32_t* group,
                                     const uint8_t* placement, int E, int M, float theta,
                                     float qbar, const double* F, const double* B,
                                     const double* tau, double z, double c, double omega_T,
                                     double omega_Q, void* tables, size_t tables_bytes_,
                                     ordermoe_stream_t stream) {
  if (!sim || !group || !placement || !F || !B || !tau || !tables)
    return fail(ORDERMOE_ERR_INVALID_ARG, "build_tables: null pointer");
  if (E <= 0 || E > ORDERMOE_MAX_EXPERTS || M <= 0 || M > ORDERMOE_MAX_SERVERS)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "build_tables: need 1 <= E <= 64, 1 <= M <= 32");
  if (tables_bytes_ < om::tables_bytes(E, M))
    return fail(ORDERMOE_ERR_INVALID_ARG, "build_tables: tables buffer too small");
  if (!(qbar >= 0.0f)) return fail(ORDERMOE_ERR_INVALID_ARG, "build_tables: qbar must be >= 0");
  if (!(c > 0.0) || !(z >= 0.0) || !(omega_T >= 0.0) || !(omega_Q >= 0.0))
    return fail(ORDERMOE_ERR_INVALID_ARG, "build_tables: need c > 0, z >= 0, omega >= 0");
  if ((reinterpret_cast<uintptr_t>(tables) & 15u) != 0)
    return fail(ORDERMOE_ERR_INVALID_ARG, "build_tables: tables must be 16-byte aligned");
  build_tables_kernel<<<1, 256, 0, stream>>>(sim, group, placement, E, M, theta, qbar, F, B, tau,
                                             z, c, omega_T, omega_Q,
                                             static_cast<uint8_t*>(tables));
  OM_LAUNCHED("build_tables_kernel");
  return ORDERMOE_OK;
}

extern "C" int ordermoe_route_select(const uint16_t* X, const uint16_t* W_r, const float* logits_in,
                                     int T, int E, int d, int k, int renorm, const void* tables,
                                     size_t tables_bytes_, const uint8_t* home, uint8_t* loc,
                                     float* qhat, float* logits_out, int32_t* topk_idx,
                                     float* topk_w, int32_t* chosen_expert,
                                     uint8_t* chosen_server, uint8_t* kind, int32_t* counters,
                                     ordermoe_stream_t stream) {
  if (T < 0) return fail(ORDERMOE_ERR_INVALID_ARG, "route_select: T < 0");
  if (E <= 0 || E > ORDERMOE_MAX_EXPERTS || k <= 0 || k > ORDERMOE_MAX_TOPK || k > E)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "route_select: need 1 <= k <= min(E, 8), E <= 64");
  if (!tables || !home || !topk_idx || !topk_w || !chosen_expert || !chosen_server || !kind)
    return fail(ORDERMOE_ERR_INVALID_ARG, "route_select: null pointer");
  if ((loc == nullptr) != (qhat == nullptr))
    return fail(ORDERMOE_ERR_INVALID_ARG, "route_select: give both loc and qhat, or neither");
  if (logits_in == nullptr) {
    if (!X || !W_r) return fail(ORDERMOE_ERR_INVALID_ARG, "route_select: X/W_r null without logits_in");
    if (d <= 0 || d % 8 != 0)
      return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "route_select: d must be a positive multiple of 8");
    if (!aligned16(X) || !aligned16(W_r))
      return fail(ORDERMOE_ERR_INVALID_ARG, "route_select: X and W_r must be 16-byte aligned");
  }
  if (tables_bytes_ < 64) return fail(ORDERMOE_ERR_INVALID_ARG, "route_select: tables too small");
  if (T == 0) return ORDERMOE_OK;
  // The table header (E, M) is on the device; E must match. Check the size
  // against the largest M so that a wrong buffer is caught early.
  if (tables_bytes_ < om::tables_bytes(E, 1))
    return fail(ORDERMOE_ERR_INVALID_ARG, "route_select: tables buffer smaller than E needs");
  const int threads = 256;
  const int per_block = threads / 32;
  int blocks = (T + per_block - 1) / per_block;
  // Stage W_r in shared memory when it fits in 96 KB; the grid is then a few
  // persistent blocks per SM so that each block loads it once.
  const size_t tab_bytes = sizeof(float) * ((2 * E * E + 3) & ~3);
  const size_t w_bytes = (size_t)E * d * 2;
  const int stage_w = (logits_in == nullptr && w_bytes <= 96 * 1024) ? 1 : 0;
  const int cap = num_sms() * (stage_w ? 2 : 8);
  if (blocks > cap) blocks = cap;
  const size_t dyn = tab_bytes + (stage_w ? w_bytes : 0);
  const uint8_t* tb = static_cast<const uint8_t*>(tables);
#define OM_RS_LAUNCH(EM)                                                                        \
  do {                                                                                          \
    cudaFuncSetAttribute(route_select_kernel<EM>, cudaFuncAttributeMaxDynamicSharedMemorySize,  \
                         (int)dyn);                                                             \
    route_select_kernel<EM><<<blocks, threads, dyn, stream>>>(                                  \
        X, W_r, logits_in, T, E, d, k, renorm, tb, home, loc, qhat, logits_out, topk_idx,       \
        topk_w, chosen_expert, chosen_server, kind, counters, stage_w);                         \
  } while (0)
  if (E <= 8) OM_RS_LAUNCH(8);
  else if (E <= 16) OM_RS_LAUNCH(16);
  else if (E <= 32) OM_RS_LAUNCH(32);
  else OM_RS_LAUNCH(64);
#undef OM_RS_LAUNCH
  OM_LAUNCHED("route_select_kernel");
  return ORDERMOE_OK;
}
