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
// Selection tables staged in shared memory (one copy per CTA).
struct SelSmem {
  uint32_t pmask[64];
  int nsub[64];
  int kind[4];
  uint8_t sublist[64 * 64];
};

// Threads t0, t0 + nt (nt >= 64) ... of the block load the layer's tables
// into shared memory. The header, masks and the first E x E entries are
// loaded before any of them is used, so that their latencies overlap; the
// E x E tables are copied with 16-byte loads where sizes and addresses
// allow.
__device__ bool load_tables_range(const uint8_t* __restrict__ tab, int E, SelSmem& sm, float* s_Q,
                                  float* s_Cq, int t0, int nt) {
  const float* gQ = reinterpret_cast<const float*>(tab + kOffQtab);
  const float* gCq = reinterpret_cast<const float*>(tab + off_cq(E));
  const int n = E * E;
  const bool vec = (n & 3) == 0 && ((reinterpret_cast<uintptr_t>(gQ) | reinterpret_cast<uintptr_t>(gCq) |
                                     reinterpret_cast<uintptr_t>(s_Q) | reinterpret_cast<uintptr_t>(s_Cq)) &
                                    15u) == 0;
  const int Eh = reinterpret_cast<const int32_t*>(tab)[1];
  const int M = reinterpret_cast<const int32_t*>(tab)[2];
  uint32_t pm = 0;
  unsigned long long sb = 0;
  if (t0 < 64) {
    pm = reinterpret_cast<const uint32_t*>(tab + kOffPmask)[t0];
    sb = reinterpret_cast<const unsigned long long*>(tab + kOffSubst)[t0];
  }
  constexpr int kFirst = 4;  // 16-byte chunks of each table a thread loads up front
  float4 q_first[kFirst], c_first[kFirst];
  if (vec) {
    const float4* q4 = reinterpret_cast<const float4*>(gQ);
    const float4* c4 = reinterpret_cast<const float4*>(gCq);
#pragma unroll
    for (int u = 0; u < kFirst; ++u) {
      const int i = t0 + u * nt;
      if (i < n / 4) {
        q_first[u] = __ldg(q4 + i);
        c_first[u] = __ldg(c4 + i);
      }
    }
  }
  if (Eh != E || M <= 0 || M > 32) {
    if (blockIdx.x == 0 && t0 == 0) report(&g_err_route, ORDERMOE_DEV_BAD_INDEX, -1);
    return false;
  }
  if (t0 < 64) {
    sm.pmask[t0] = pm;
    int cnt = 0;
    while (sb) {
      const int b = __ffsll(static_cast<long long>(sb)) - 1;
      sm.sublist[t0 * 64 + cnt++] = static_cast<uint8_t>(b);
      sb &= sb - 1;
    }
    sm.nsub[t0] = cnt;
  }
  if (vec) {
    const float4* q4 = reinterpret_cast<const float4*>(gQ);
    const float4* c4 = reinterpret_cast<const float4*>(gCq);
#pragma unroll
    for (int u = 0; u < kFirst; ++u) {
      const int i = t0 + u * nt;
      if (i < n / 4) {
        reinterpret_cast<float4*>(s_Q)[i] = q_first[u];
        reinterpret_cast<float4*>(s_Cq)[i] = c_first[u];
      }
    }
#pragma unroll 4
    for (int i = t0 + kFirst * nt; i < n / 4; i += nt) {
      const float4 x = __ldg(q4 + i), y = __ldg(c4 + i);
      reinterpret_cast<float4*>(s_Q)[i] = x;
      reinterpret_cast<float4*>(s_Cq)[i] = y;
    }
  } else {
#pragma unroll 4
    for (int i = t0; i < n; i += nt) {
      s_Q[i] = gQ[i];
      s_Cq[i] = gCq[i];
    }
  }
  for (int i = t0; i < 4; i += nt) sm.kind[i] = 0;
  return true;
}

// Loads the layer's tables into shared memory (whole block). Returns false
// if the header does not match E (reported once).
__device__ bool load_tables(const uint8_t* __restrict__ tab, int E, SelSmem& sm, float* s_Q,
                            float* s_Cq) {
  return load_tables_range(tab, E, sm, s_Q, s_Cq, threadIdx.x, blockDim.x);  // blockDim.x >= 64
}

// The delay table A[a][s][m] of Eq. 38 (M^3 floats) is read once per
// candidate (expert, server) of every slot, so the selection keeps it in
// shared memory when it has at most kDelayStage entries (M <= 16);
// larger tables stay in global memory. Threads t0, t0 + nt, ... copy it;
// every thread gets the same pointer back, the one the selection reads.
constexpr int kDelayStage = 4096;
__device__ const float* load_delay_range(const uint8_t* __restrict__ tab, int E, float* s_A,
                                         int t0, int nt) {
  const int M = reinterpret_cast<const int32_t*>(tab)[2];
  const float* gA = reinterpret_cast<const float*>(tab + off_a(E));
  if (M <= 0 || M > 16) return gA;
  const int n = M * M * M;
  for (int i = t0; i < n; i += nt) s_A[i] = gA[i];
  return s_A;
}

// Look-ahead context (Eqs. 41-43): the tables of the next layers follow the
// current layer's at a fixed byte stride; P holds P_l .. P_{l+H-2}.
struct Lookahead {
  int H;                 // horizon; 1 = myopic (Phi = 0)
  size_t stride;         // bytes between consecutive layers' tables
  const float* P;        // [H-1][E][E]
  int staged;            // lookahead_select_kernel copies layers l+1.. and P to shared memory
  int topk_only;         // H = 1 with many experts: the router writes the targets and weights,
                         // select_lanes_kernel selects
};

// A plain (generic) load: the look-ahead reads the next layers' tables either
// from global memory or from the kernel's shared-memory copy of them.
template <class T>
__device__ __forceinline__ T ldt(const T* p) {
  return *p;
}

// Cost-to-go of Eq. 42 with D future layers, from server m after executing
// expert kx with accumulated loss qacc: sum over next targets k' (ascending)
// of P(kx -> k') times the cheapest feasible (m', k'') of the next layer
// (Eq. 40 from server m; a single target, no distinct-expert rule), each
// plus its own cost-to-go. Every product and sum is one rounded fp32
// operation, so the value is reproducible bit for bit.
template <int D>
__device__ float lookahead_phi(const uint8_t* __restrict__ tnext, size_t stride,
                               const float* __restrict__ P, int E, int M, int a, int m, int kx,
                               float qacc, float qbar) {
  const float* Q1 = reinterpret_cast<const float*>(tnext + kOffQtab);
  const float* C1 = reinterpret_cast<const float*>(tnext + off_cq(E));
  const float* A1 = reinterpret_cast<const float*>(tnext + off_a(E));
  const uint32_t* pm1 = reinterpret_cast<const uint32_t*>(tnext + kOffPmask);
  const unsigned long long* sb1 = reinterpret_cast<const unsigned long long*>(tnext + kOffSubst);
  float acc = 0.0f;
  for (int kt = 0; kt < E; ++kt) {
    const float p = ldt(P + (size_t)kx * E + kt);
    if (p == 0.0f) continue;
    float best = INFINITY;
    unsigned long long cand = ldt(sb1 + kt) | (1ull << kt);  // substitutes and the target
    while (cand) {
      const int kk = __ffsll(static_cast<long long>(cand)) - 1;
      cand &= cand - 1;
      const bool exact = (kk == kt);
      float cq = 0.0f, q2 = qacc;
      if (!exact) {
        const float qk = ldt(Q1 + kt * E + kk);
        if (!(__fadd_rn(qacc, qk) <= qbar)) continue;
        q2 = __fadd_rn(qacc, qk);
        cq = ldt(C1 + kt * E + kk);
      }
      uint32_t pm = ldt(pm1 + kk);
      while (pm) {
        const int m2 = __ffs(pm) - 1;
        pm &= pm - 1;
        float c = __fadd_rn(ldt(A1 + ((size_t)a * M + m) * M + m2), cq);
        if (D > 1)
          c = __fadd_rn(c, lookahead_phi<(D > 1 ? D - 1 : 1)>(tnext + stride, stride, P + E * E, E,
                                                              M, a, m2, kk, q2, qbar));
        best = fminf(best, c);
      }
    }
    acc = __fadd_rn(acc, __fmul_rn(p, best));
  }
  return acc;
}

__device__ __forceinline__ float lookahead_cost(const Lookahead& la, const uint8_t* tab, int E,
                                                int M, int a, int m, int kx, float qacc,
                                                float qbar) {
  switch (la.H) {
    case 2: return lookahead_phi<1>(tab + la.stride, la.stride, la.P, E, M, a, m, kx, qacc, qbar);
    case 3: return lookahead_phi<2>(tab + la.stride, la.stride, la.P, E, M, a, m, kx, qacc, qbar);
    case 4: return lookahead_phi<3>(tab + la.stride, la.stride, la.P, E, M, a, m, kx, qacc, qbar);
    default: return 0.0f;
  }
}

// A token's logits in shared memory as 16-byte chunks: chunk c holds
// logits 4c .. 4c + 3 (-inf past E), at p[128 c] (one thread's column of a
// [chunk][128 tokens] array, so the 32 tokens of a warp read consecutive
// chunks: no bank conflicts).
struct ColLogits {
  const float4* p;
  __device__ __forceinline__ float4 chunk(int c) const { return p[c * 128]; }
};

// The KN largest of the token's nc chunks of logits by (logit desc, index
// asc) into v[0..KN), ix[0..KN), as a sorted list built by inserting the
// logits in index order: logit e goes to the first position whose value it
// exceeds, so an equal value stays behind the earlier index, and the entries
// from that position on move down one. The positions it exceeds form a
// suffix of the list (g[p] implies g[p+1]), which makes every position one
// select of its own value, the new logit or its predecessor; positions
// p >= e are still empty when logit e arrives. The list stays in registers
// (compile-time positions), nothing branches inside a chunk, and the loop
// over chunks keeps the code short (a long unrolled form stalled on
// instruction fetch). The -inf logits past E go behind every real one, so
// the first k <= E entries are real. Returns whether a logit was NaN.
template <int KN, class Src>
__device__ __forceinline__ bool topk_list(const Src& src, int nc, float (&v)[ORDERMOE_MAX_TOPK],
                                          int (&ix)[ORDERMOE_MAX_TOPK]) {
#pragma unroll
  for (int p = 0; p < ORDERMOE_MAX_TOPK; ++p) {
    v[p] = -INFINITY;
    ix[p] = -1;
  }
  bool nan = false;
#pragma unroll 1
  for (int c4 = 0; c4 < nc; ++c4) {
    const float4 x4 = src.chunk(c4);
    const float xs[4] = {x4.x, x4.y, x4.z, x4.w};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const float c = xs[u];
      const int e = 4 * c4 + u;
      nan |= isnan(c);
      bool g[KN];
#pragma unroll
      for (int p = 0; p < KN; ++p) g[p] = (p >= e) | (c > v[p]);
#pragma unroll
      for (int p = KN - 1; p >= 1; --p) {
        const float tv = g[p] ? c : v[p];
        const int ti = g[p] ? e : ix[p];
        v[p] = g[p - 1] ? v[p - 1] : tv;
        ix[p] = g[p - 1] ? ix[p - 1] : ti;
      }
      v[0] = g[0] ? c : v[0];
      ix[0] = g[0] ? e : ix[0];
    }
  }
  return nan;
}

// One token: softmax over E, top-k, then Alg. 2 (H = 1) per slot in rank
// order (Eqs. 36-44). src gives the logits in 16-byte chunks (ColLogits).
// The caller loads the token's home a, location s (Eq. 36: a on the first
// layer) and accumulated loss q. Atab is the delay table of Eq. 38, in
// shared or global memory. The argmin of Eq. 43 packs (fp32 cost bits,
// substitute, away, server, expert) into a 64-bit key and keeps the
// smallest; costs are never negative, so the bit pattern orders them like
// the values.
template <class Src>
__device__ __forceinline__ void select_token(
    int t, const Src& src, int E, int k, int renorm, int M, float qbar,
    const float* Atab, const uint8_t* __restrict__ tab, const Lookahead& la,
    const SelSmem& sm, const float* s_Q, const float* s_Cq, int a, int s, float q,
    uint8_t* __restrict__ loc, float* __restrict__ qhat,
    int32_t* __restrict__ topk_idx, float* __restrict__ topk_w, int32_t* __restrict__ chosen_expert,
    uint8_t* __restrict__ chosen_server, uint8_t* __restrict__ kind_out, int (&kind_count)[4],
    bool topk_only = false) {
  // top-k by (logit desc, index asc): a sorted list of 2, 4, 6 or 8 >= k
  float vtop[ORDERMOE_MAX_TOPK];
  int itop[ORDERMOE_MAX_TOPK];
  const int nc = (E + 3) / 4;
  bool nan;
  if (k <= 2) nan = topk_list<2>(src, nc, vtop, itop);
  else if (k <= 4) nan = topk_list<4>(src, nc, vtop, itop);
  else if (k <= 6) nan = topk_list<6>(src, nc, vtop, itop);
  else nan = topk_list<8>(src, nc, vtop, itop);
  if (nan) {
    report(&g_err_route, ORDERMOE_DEV_NAN_LOGIT, t);
    for (int j = 0; j < k; ++j) {  // no targets: a later pass skips this token
      topk_idx[(size_t)t * k + j] = -1;
      topk_w[(size_t)t * k + j] = 0.0f;
    }
    return;
  }
  // softmax over all E in fp32, summed in index order (the maximum is the
  // list's head; the -inf logits past E add exact zeros after the real
  // terms); gate weights of the k slots
  const float lmax = vtop[0];
  float denom = 0.0f;
#pragma unroll 1
  for (int c4 = 0; c4 < nc; ++c4) {
    const float4 x4 = src.chunk(c4);
    denom += expf(x4.x - lmax);
    denom += expf(x4.y - lmax);
    denom += expf(x4.z - lmax);
    denom += expf(x4.w - lmax);
  }
  float wsel[ORDERMOE_MAX_TOPK];
  float ssel = 0.0f;
#pragma unroll
  for (int j = 0; j < ORDERMOE_MAX_TOPK; ++j)
    if (j < k) {
      wsel[j] = expf(vtop[j] - lmax) / denom;
      ssel += wsel[j];
    }
  int idx[ORDERMOE_MAX_TOPK];
  unsigned long long used_targets = 0;
#pragma unroll
  for (int j = 0; j < ORDERMOE_MAX_TOPK; ++j) {
    idx[j] = itop[j];
    if (j < k) {
      topk_idx[(size_t)t * k + j] = itop[j];
      topk_w[(size_t)t * k + j] = renorm ? wsel[j] / ssel : wsel[j];
      used_targets |= 1ull << itop[j];
    }
  }
  if (topk_only) return;
  // selection
  if (a >= M || s >= M) {
    report(&g_err_route, ORDERMOE_DEV_BAD_INDEX, t);
    return;
  }
  const float* Aas = Atab + (a * M + s) * M;
  unsigned long long taken = used_targets;
  int first_server = s;
  for (int j = 0; j < k; ++j) {
    const int r = idx[j];
    const int nsub = sm.nsub[r];
    unsigned long long best = ~0ull;
    for (int ki = 0; ki <= nsub; ++ki) {
      const int kk = (ki == 0) ? r : sm.sublist[r * 64 + ki - 1];
      const bool sub = (ki != 0);
      float cq = 0.0f, qn = q;
      if (sub) {
        if ((taken >> kk) & 1ull) continue;
        if (!(__fadd_rn(q, s_Q[r * E + kk]) <= qbar)) continue;  // Eq. 40 budget
        cq = s_Cq[r * E + kk];
        qn = __fadd_rn(q, s_Q[r * E + kk]);
      }
      uint32_t pm = sm.pmask[kk];
      while (pm) {
        const int m = __ffs(pm) - 1;
        pm &= pm - 1;
        float cost = __fadd_rn(Aas[m], cq);
        if (la.H > 1) cost = __fadd_rn(cost, lookahead_cost(la, tab, E, M, a, m, kk, qn, qbar));
        const unsigned long long key =
            (static_cast<unsigned long long>(__float_as_uint(cost)) << 32) |
            (static_cast<unsigned long long>(sub ? 1u : 0u) << 31) |
            (static_cast<unsigned long long>(m != s ? 1u : 0u) << 30) |
            (static_cast<unsigned long long>(m) << 8) | static_cast<unsigned long long>(kk);
        best = key < best ? key : best;
      }
    }
    int kstar, mstar, kd;
    if (best == ~0ull) {
      report(&g_err_route, ORDERMOE_DEV_NO_CANDIDATE, t);
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
    chosen_expert[(size_t)t * k + j] = kstar;
    chosen_server[(size_t)t * k + j] = static_cast<uint8_t>(mstar);
    kind_out[(size_t)t * k + j] = static_cast<uint8_t>(kd);
    if (kd == 0) ++kind_count[0];  // constant indices: kind_count[] stays in registers
    else if (kd == 1) ++kind_count[1];
    else if (kd == 2) ++kind_count[2];
    else ++kind_count[3];
  }
  if (loc != nullptr) {
    loc[t] = static_cast<uint8_t>(first_server);
    qhat[t] = q;
  }
}

__device__ __forceinline__ void flush_kind_counts(SelSmem& sm, const int (&kind_count)[4],
                                                  int32_t* counters) {
  if (counters == nullptr) return;
  for (int i = 0; i < 4; ++i)
    if (kind_count[i]) atomicAdd(&sm.kind[i], kind_count[i]);
}

// Selection from given logits: one thread per token.
template <int EMAX>
__global__ void __launch_bounds__(128) select_kernel(
    const float* __restrict__ logits_in, int T, int E, int k, int renorm,
    const uint8_t* __restrict__ tab, const uint8_t* __restrict__ home, uint8_t* __restrict__ loc,
    float* __restrict__ qhat, float* __restrict__ logits_out, int32_t* __restrict__ topk_idx,
    float* __restrict__ topk_w, int32_t* __restrict__ chosen_expert,
    uint8_t* __restrict__ chosen_server, uint8_t* __restrict__ kind_out,
    int32_t* __restrict__ counters, Lookahead la) {
  pdl_trigger();  // launched with launch_pdl: no global access before pdl_wait
  pdl_wait();
  __shared__ SelSmem sm;
  extern __shared__ __align__(16) float s_dyn[];
  float4* s_lg = reinterpret_cast<float4*>(s_dyn);  // [EMAX / 4][128] chunks of logits
  float* s_Q = s_dyn + EMAX * 128;
  float* s_Cq = s_Q + E * E;
  const int t = blockIdx.x * blockDim.x + threadIdx.x;
  // the token's state first: its loads overlap the tables'
  int a = 0, sl = 0;
  float q0 = 0.0f;
  if (t < T && la.H == 1) {
    a = home[t];
    sl = (loc != nullptr) ? loc[t] : a;  // no state given: first layer (Eq. 36)
    q0 = (qhat != nullptr) ? qhat[t] : 0.0f;
  }
  if (!load_tables(tab, E, sm, s_Q, s_Cq)) return;
  const float* Atab = load_delay_range(tab, E, s_Cq + E * E, threadIdx.x, blockDim.x);
  __syncthreads();
  const int M = reinterpret_cast<const int32_t*>(tab)[2];
  const float qbar = reinterpret_cast<const float*>(tab)[5];
  int kind_count[4] = {0, 0, 0, 0};
  if (t < T) {
    float lg[EMAX];
#pragma unroll
    for (int e = 0; e < EMAX; ++e) lg[e] = (e < E) ? logits_in[(size_t)t * E + e] : -INFINITY;
    if (logits_out != nullptr) {
#pragma unroll
      for (int e = 0; e < EMAX; ++e)  // constant indices keep lg[] in registers
        if (e < E) logits_out[(size_t)t * E + e] = lg[e];
    }
#pragma unroll
    for (int c = 0; c < EMAX; c += 4)
      s_lg[(c / 4) * 128 + threadIdx.x] = make_float4(lg[c], lg[c + 1], lg[c + 2], lg[c + 3]);
    select_token(t, ColLogits{s_lg + threadIdx.x}, E, k, renorm, M, qbar, Atab, tab, la, sm, s_Q,
                 s_Cq, a, sl, q0, loc, qhat, topk_idx, topk_w, chosen_expert, chosen_server,
                 kind_out, kind_count, la.H > 1);
  }
  flush_kind_counts(sm, kind_count, counters);
  __syncthreads();
  if (counters != nullptr && threadIdx.x < 4 && sm.kind[threadIdx.x])
    atomicAdd(&counters[threadIdx.x], sm.kind[threadIdx.x]);
}

// ---------------------------------------------------------------------------
// Alg. 2 with H = 1 from the targets topk_idx, eight lanes per token: for
// each slot the lanes split the target and its substitutes (lane j takes
// candidates j, j + 8, ... of the list), each keeps the smallest 64-bit key
// of select_token (cost bits, substitute, away, server, expert: a total
// order, so the minimum over any split is the same), and three butterfly
// steps over the eight lanes give the slot's argmin to all of them; they
// then update the taken set and the loss identically. Used for many experts,
// where one thread per token walks a long serial chain of candidates.
constexpr int kLaneTokens = 4;   // tokens per warp (eight lanes each)
constexpr int kLaneThreads = 256;

__global__ void __launch_bounds__(kLaneThreads) select_lanes_kernel(
    const int32_t* __restrict__ topk_idx, int T, int E, int k, const uint8_t* __restrict__ tab,
    const uint8_t* __restrict__ home, uint8_t* __restrict__ loc, float* __restrict__ qhat,
    int32_t* __restrict__ chosen_expert, uint8_t* __restrict__ chosen_server,
    uint8_t* __restrict__ kind_out, int32_t* __restrict__ counters) {
  pdl_trigger();  // launched with launch_pdl: no global access before pdl_wait
  pdl_wait();
  __shared__ SelSmem sm;
  extern __shared__ __align__(16) float s_dyn[];
  float* s_Q = s_dyn;
  float* s_Cq = s_dyn + E * E;
  if (!load_tables(tab, E, sm, s_Q, s_Cq)) return;
  // the delay table stays in global memory here: staging it took longer
  // than the reads it saves (one per candidate, eight lanes at a time)
  const float* Atab = reinterpret_cast<const float*>(tab + off_a(E));
  __syncthreads();
  const int M = reinterpret_cast<const int32_t*>(tab)[2];
  const float qbar = reinterpret_cast<const float*>(tab)[5];
  const int lane = threadIdx.x & 31;
  const int sub = lane & 7;       // lane within the token's group of eight
  const int grp = lane >> 3;
  const int warps_total = gridDim.x * (kLaneThreads / 32);
  int kind_count[4] = {0, 0, 0, 0};
  for (int base = (blockIdx.x * (kLaneThreads / 32) + (threadIdx.x >> 5)) * kLaneTokens; base < T;
       base += warps_total * kLaneTokens) {
    const int t = base + grp;
    // every lane runs every slot (the butterflies need the whole warp);
    // inactive tokens (past T, a NaN token's -1 targets, bad servers) write nothing
    bool active = t < T;
    // the token's state and targets, loaded together
    int a = 0, s = 0;
    float q = 0.0f;
    if (active) {
      a = home[t];
      s = (loc != nullptr) ? loc[t] : a;
      q = (qhat != nullptr) ? qhat[t] : 0.0f;
    }
    int idx[ORDERMOE_MAX_TOPK];
    unsigned long long taken = 0;
#pragma unroll
    for (int j = 0; j < ORDERMOE_MAX_TOPK; ++j) idx[j] = (j < k && active) ? topk_idx[(size_t)t * k + j] : 0;
#pragma unroll
    for (int j = 0; j < ORDERMOE_MAX_TOPK; ++j)
      if (j < k && active) {
        if (idx[j] < 0 || idx[j] >= E) active = false;
        else taken |= 1ull << idx[j];
      }
    if (active && (a >= M || s >= M)) {
      if (sub == 0) report(&g_err_route, ORDERMOE_DEV_BAD_INDEX, t);
      active = false;
    }
    const float* Aas = Atab + (active ? (a * M + s) * M : 0);
    int first_server = s;
#pragma unroll
    for (int j = 0; j < ORDERMOE_MAX_TOPK; ++j) {
      if (j >= k) break;  // k is the same for every lane
      const int r = idx[j];
      const int nsub = active ? sm.nsub[r] : -1;
      unsigned long long best = ~0ull;
      for (int ki = sub; ki <= nsub; ki += 8) {
        const int kk = (ki == 0) ? r : sm.sublist[r * 64 + ki - 1];
        const bool issub = (ki != 0);
        float cq = 0.0f;
        if (issub) {
          if ((taken >> kk) & 1ull) continue;
          if (!(__fadd_rn(q, s_Q[r * E + kk]) <= qbar)) continue;  // Eq. 40 budget
          cq = s_Cq[r * E + kk];
        }
        uint32_t pm = sm.pmask[kk];
        while (pm) {
          const int m = __ffs(pm) - 1;
          pm &= pm - 1;
          const float cost = __fadd_rn(Aas[m], cq);
          const unsigned long long key =
              (static_cast<unsigned long long>(__float_as_uint(cost)) << 32) |
              (static_cast<unsigned long long>(issub ? 1u : 0u) << 31) |
              (static_cast<unsigned long long>(m != s ? 1u : 0u) << 30) |
              (static_cast<unsigned long long>(m) << 8) | static_cast<unsigned long long>(kk);
          best = key < best ? key : best;
        }
      }
#pragma unroll
      for (int o = 4; o > 0; o >>= 1) {
        const unsigned long long other = __shfl_xor_sync(0xffffffffu, best, o);
        best = other < best ? other : best;
      }
      if (!active) continue;
      int kstar, mstar, kd;
      if (best == ~0ull) {
        if (sub == 0) report(&g_err_route, ORDERMOE_DEV_NO_CANDIDATE, t);
        kstar = r; mstar = s; kd = 0;
      } else {
        kstar = static_cast<int>(best & 0xFFu);
        mstar = static_cast<int>((best >> 8) & 0xFFu);
        const int bsub = static_cast<int>((best >> 31) & 1u);
        const int away = static_cast<int>((best >> 30) & 1u);
        kd = 2 * away + bsub;
        if (bsub) {
          taken |= 1ull << kstar;
          q = __fadd_rn(q, s_Q[r * E + kstar]);
        }
      }
      if (j == 0) first_server = mstar;
      if (sub == 0) {
        chosen_expert[(size_t)t * k + j] = kstar;
        chosen_server[(size_t)t * k + j] = static_cast<uint8_t>(mstar);
        kind_out[(size_t)t * k + j] = static_cast<uint8_t>(kd);
        if (kd == 0) ++kind_count[0];  // constant indices: kind_count[] stays in registers
        else if (kd == 1) ++kind_count[1];
        else if (kd == 2) ++kind_count[2];
        else ++kind_count[3];
      }
    }
    if (active && sub == 0 && loc != nullptr) {
      loc[t] = static_cast<uint8_t>(first_server);
      qhat[t] = q;
    }
  }
  flush_kind_counts(sm, kind_count, counters);
  __syncthreads();
  if (counters != nullptr && threadIdx.x < 4 && sm.kind[threadIdx.x])
    atomicAdd(&counters[threadIdx.x], sm.kind[threadIdx.x]);
}

// ---------------------------------------------------------------------------
// Alg. 2 with horizon H > 1 (Eq. 43), one block per token, from the targets
// topk_idx. For each slot the block lists the slot's candidates (expert,
// server) in shared memory, then every thread takes (candidate, next target
// k') items: the term P(k -> k') * min(...) of Eq. 42, with the deeper levels
// of the recursion serial in the thread. Each candidate's terms are then
// added in ascending k' (skipping P = 0, as the serial definition does), so
// Phi is the same fp32 value; the argmin key is reduced with atomicMin.
template <int D>
__device__ __forceinline__ float phi_term(const uint8_t* __restrict__ tnext, size_t stride,
                                          const float* __restrict__ P, int E, int M, int a, int m,
                                          int kx, int kt, float qacc, float qbar) {
  // the k' = kt term of lookahead_phi<D> (0 when P = 0)
  const float p = ldt(P + (size_t)kx * E + kt);
  if (p == 0.0f) return 0.0f;
  const float* Q1 = reinterpret_cast<const float*>(tnext + kOffQtab);
  const float* C1 = reinterpret_cast<const float*>(tnext + off_cq(E));
  const float* A1 = reinterpret_cast<const float*>(tnext + off_a(E));
  const uint32_t* pm1 = reinterpret_cast<const uint32_t*>(tnext + kOffPmask);
  const unsigned long long* sb1 = reinterpret_cast<const unsigned long long*>(tnext + kOffSubst);
  float best = INFINITY;
  unsigned long long cand = ldt(sb1 + kt) | (1ull << kt);
  while (cand) {
    const int kk = __ffsll(static_cast<long long>(cand)) - 1;
    cand &= cand - 1;
    const bool exact = (kk == kt);
    float cq = 0.0f, q2 = qacc;
    if (!exact) {
      const float qk = ldt(Q1 + kt * E + kk);
      if (!(__fadd_rn(qacc, qk) <= qbar)) continue;
      q2 = __fadd_rn(qacc, qk);
      cq = ldt(C1 + kt * E + kk);
    }
    uint32_t pm = ldt(pm1 + kk);
    while (pm) {
      const int m2 = __ffs(pm) - 1;
      pm &= pm - 1;
      float c = __fadd_rn(ldt(A1 + ((size_t)a * M + m) * M + m2), cq);
      if (D > 1)
        c = __fadd_rn(c, lookahead_phi<(D > 1 ? D - 1 : 1)>(tnext + stride, stride, P + E * E, E,
                                                            M, a, m2, kk, q2, qbar));
      best = fminf(best, c);
    }
  }
  return __fmul_rn(p, best);
}

// H = 3: the term of Eq. 42 with the deepest cost-to-go Phi^(1)(m2, k2, q2)
// read from a per-token table U[m2][k2] whenever no budget check of that level
// can fail: U was evaluated with q2 = 0, and with Qmax[k2] the largest loss of
// a substitute that level can consider (targets k' with P(k2 -> k') != 0),
// fadd(q2, Qmax[k2]) <= Qbar means every check passes for q2 as for 0 (fadd
// is monotone and q2 >= 0), so the value is the same; otherwise it is
// evaluated directly.
__device__ __forceinline__ float phi_term2_memo(const uint8_t* __restrict__ tnext, size_t stride,
                                                const float* __restrict__ P, int E, int M, int a,
                                                int m, int kx, int kt, float qacc, float qbar,
                                                const float* U, const float* qmax1) {
  const float p = ldt(P + (size_t)kx * E + kt);
  if (p == 0.0f) return 0.0f;
  const float* Q1 = reinterpret_cast<const float*>(tnext + kOffQtab);
  const float* C1 = reinterpret_cast<const float*>(tnext + off_cq(E));
  const float* A1 = reinterpret_cast<const float*>(tnext + off_a(E));
  const uint32_t* pm1 = reinterpret_cast<const uint32_t*>(tnext + kOffPmask);
  const unsigned long long* sb1 = reinterpret_cast<const unsigned long long*>(tnext + kOffSubst);
  float best = INFINITY;
  unsigned long long cand = ldt(sb1 + kt) | (1ull << kt);
  while (cand) {
    const int kk = __ffsll(static_cast<long long>(cand)) - 1;
    cand &= cand - 1;
    const bool exact = (kk == kt);
    float cq = 0.0f, q2 = qacc;
    if (!exact) {
      const float qk = ldt(Q1 + kt * E + kk);
      if (!(__fadd_rn(qacc, qk) <= qbar)) continue;
      q2 = __fadd_rn(qacc, qk);
      cq = ldt(C1 + kt * E + kk);
    }
    const bool free = __fadd_rn(q2, qmax1[kk]) <= qbar;
    uint32_t pm = ldt(pm1 + kk);
    while (pm) {
      const int m2 = __ffs(pm) - 1;
      pm &= pm - 1;
      const float phi1 = free ? U[m2 * E + kk]
                              : lookahead_phi<1>(tnext + stride, stride, P + E * E, E, M, a, m2, kk,
                                                 q2, qbar);
      const float c = __fadd_rn(__fadd_rn(ldt(A1 + ((size_t)a * M + m) * M + m2), cq), phi1);
      best = fminf(best, c);
    }
  }
  return __fmul_rn(p, best);
}

// An order-preserving map of fp32 onto uint32 (the minimum of the keys is the
// key of the minimum), so that partial minima can be joined with atomicMin.
__device__ __forceinline__ uint32_t min_key(float x) {
  const uint32_t b = __float_as_uint(x);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float from_min_key(uint32_t key) {
  return __uint_as_float((key & 0x80000000u) ? (key & 0x7FFFFFFFu) : ~key);
}

// Pairs (k'', m2) of phi_term2_memo whose Phi^(1) is not in U, listed for a
// parallel evaluation: code = item << 16 | m2 << 8 | k'' (item: the
// (candidate, k') term they belong to), A(a, m, m2) + Cq, and the loss q2.
constexpr int kLaSlow = 512;         // listed pairs per pass
constexpr int kLaSlowTerms = 2048;   // their Phi^(1) terms per sub-pass
constexpr size_t kLaSlowBytes = (size_t)kLaSlow * 12 + (size_t)kLaSlowTerms * 4;
struct LaSlow {
  uint32_t* code;
  float* base;
  float* q2;
  float* terms;
};

// phi_term2_memo split in two: the minimum over the pairs whose Phi^(1) is
// read from U is returned (as a min_key), and each other pair is appended to
// the list (or, when the list is full, evaluated here). The caller joins the
// listed pairs' costs into the minimum and multiplies by P(kx -> kt); the
// minimum of a set does not depend on the order it is taken in, so the term
// is the same fp32 value.
__device__ __forceinline__ uint32_t phi_term2_split(const uint8_t* __restrict__ tnext,
                                                    size_t stride, const float* __restrict__ P,
                                                    int E, int M, int a, int m, int kx, int kt,
                                                    float qacc, float qbar, const float* U,
                                                    const float* qmax1, int item,
                                                    const LaSlow& slow, int* ns) {
  const float* Q1 = reinterpret_cast<const float*>(tnext + kOffQtab);
  const float* C1 = reinterpret_cast<const float*>(tnext + off_cq(E));
  const float* A1 = reinterpret_cast<const float*>(tnext + off_a(E));
  const uint32_t* pm1 = reinterpret_cast<const uint32_t*>(tnext + kOffPmask);
  const unsigned long long* sb1 = reinterpret_cast<const unsigned long long*>(tnext + kOffSubst);
  float best = INFINITY;
  unsigned long long cand = ldt(sb1 + kt) | (1ull << kt);
  while (cand) {
    const int kk = __ffsll(static_cast<long long>(cand)) - 1;
    cand &= cand - 1;
    const bool exact = (kk == kt);
    float cq = 0.0f, q2 = qacc;
    if (!exact) {
      const float qk = ldt(Q1 + kt * E + kk);
      if (!(__fadd_rn(qacc, qk) <= qbar)) continue;
      q2 = __fadd_rn(qacc, qk);
      cq = ldt(C1 + kt * E + kk);
    }
    const bool free = __fadd_rn(q2, qmax1[kk]) <= qbar;
    uint32_t pm = ldt(pm1 + kk);
    while (pm) {
      const int m2 = __ffs(pm) - 1;
      pm &= pm - 1;
      const float base = __fadd_rn(ldt(A1 + ((size_t)a * M + m) * M + m2), cq);
      if (free) {
        best = fminf(best, __fadd_rn(base, U[m2 * E + kk]));
        continue;
      }
      const int e = atomicAdd(ns, 1);
      if (e < kLaSlow) {
        slow.code[e] = (static_cast<uint32_t>(item) << 16) | (static_cast<uint32_t>(m2) << 8) |
                       static_cast<uint32_t>(kk);
        slow.base[e] = base;
        slow.q2[e] = q2;
      } else {
        best = fminf(best, __fadd_rn(base, lookahead_phi<1>(tnext + stride, stride, P + E * E, E,
                                                            M, a, m2, kk, q2, qbar)));
      }
    }
  }
  return min_key(best);
}

// lookahead_phi<2> with its deepest level read from U / qmax1 as in
// phi_term2_memo (the same fp32 operations in the same order).
__device__ float lookahead_phi2_memo(const uint8_t* __restrict__ tnext, size_t stride,
                                     const float* __restrict__ P, int E, int M, int a, int m,
                                     int kx, float qacc, float qbar, const float* U,
                                     const float* qmax1) {
  float acc = 0.0f;
  for (int kt = 0; kt < E; ++kt) {
    if (ldt(P + (size_t)kx * E + kt) == 0.0f) continue;
    acc = __fadd_rn(acc, phi_term2_memo(tnext, stride, P, E, M, a, m, kx, kt, qacc, qbar, U, qmax1));
  }
  return acc;
}

// H = 4: the term of Eq. 42 with Phi^(2)(m2, k2, q2) read from a per-token
// table U2[m2][k2] (evaluated with q2 = 0) whenever no budget check inside it
// can fail: every loss it adds at its own level is at most qmax2[k2] and every
// loss one level deeper at most qmaxL1 (losses are not negative; -inf: none),
// so fadd(q2, qmax2[k2]) <= Qbar and fadd(that, qmaxL1) <= Qbar mean every
// check passes for q2 as for 0 (fadd is monotone) and the value is the same.
// Otherwise Phi^(2) is evaluated, its deepest level again from U1 when free.
__device__ __forceinline__ float phi_term3_memo(const uint8_t* __restrict__ tnext, size_t stride,
                                                const float* __restrict__ P, int E, int M, int a,
                                                int m, int kx, int kt, float qacc, float qbar,
                                                const float* U2, const float* qmax2, float qmaxL1,
                                                const float* U1, const float* qmax1) {
  const float p = ldt(P + (size_t)kx * E + kt);
  if (p == 0.0f) return 0.0f;
  const float* Q1 = reinterpret_cast<const float*>(tnext + kOffQtab);
  const float* C1 = reinterpret_cast<const float*>(tnext + off_cq(E));
  const float* A1 = reinterpret_cast<const float*>(tnext + off_a(E));
  const uint32_t* pm1 = reinterpret_cast<const uint32_t*>(tnext + kOffPmask);
  const unsigned long long* sb1 = reinterpret_cast<const unsigned long long*>(tnext + kOffSubst);
  float best = INFINITY;
  unsigned long long cand = ldt(sb1 + kt) | (1ull << kt);
  while (cand) {
    const int kk = __ffsll(static_cast<long long>(cand)) - 1;
    cand &= cand - 1;
    const bool exact = (kk == kt);
    float cq = 0.0f, q2 = qacc;
    if (!exact) {
      const float qk = ldt(Q1 + kt * E + kk);
      if (!(__fadd_rn(qacc, qk) <= qbar)) continue;
      q2 = __fadd_rn(qacc, qk);
      cq = ldt(C1 + kt * E + kk);
    }
    const float qa = __fadd_rn(q2, qmax2[kk]);
    const float q3max = (qmax2[kk] == -INFINITY) ? q2 : qa;  // largest loss entering level 1
    const bool free = qa <= qbar && __fadd_rn(q3max, qmaxL1) <= qbar;
    uint32_t pm = ldt(pm1 + kk);
    while (pm) {
      const int m2 = __ffs(pm) - 1;
      pm &= pm - 1;
      const float phi2 = free ? U2[m2 * E + kk]
                              : lookahead_phi2_memo(tnext + stride, stride, P + E * E, E, M, a, m2,
                                                    kk, q2, qbar, U1, qmax1);
      const float c = __fadd_rn(__fadd_rn(ldt(A1 + ((size_t)a * M + m) * M + m2), cq), phi2);
      best = fminf(best, c);
    }
  }
  return __fmul_rn(p, best);
}

// tn: the tables of layer l + 1 (the deeper layers follow, stride bytes
// apart), Pn: the transitions l -> l + 1 (the deeper ones follow).
__device__ __forceinline__ float phi_term_h(int H, const uint8_t* tn, size_t stride,
                                            const float* Pn, int E, int M, int a, int m, int kx,
                                            int kt, float qacc, float qbar) {
  switch (H) {
    case 2: return phi_term<1>(tn, stride, Pn, E, M, a, m, kx, kt, qacc, qbar);
    case 3: return phi_term<2>(tn, stride, Pn, E, M, a, m, kx, kt, qacc, qbar);
    case 4: return phi_term<3>(tn, stride, Pn, E, M, a, m, kx, kt, qacc, qbar);
    default: return 0.0f;
  }
}

// Shared-memory copy of the next layers' tables and transitions for the
// look-ahead (bytes after the E x E tables and the H = 4 extras).
__host__ __device__ inline size_t la_stage_offset(int E, int H) {
  const size_t f = 2 * (size_t)E * E + (H == 4 ? 33 * (size_t)E : 0);
  return (f * sizeof(float) + 15) & ~size_t(15);
}
__host__ __device__ inline size_t la_stage_bytes(int E, int H, size_t stride) {
  return (size_t)(H - 1) * stride + (size_t)(H - 1) * E * E * sizeof(float);
}
// H = 3: the pairs listed by phi_term2_split follow the tables (and their
// shared-memory copy, when there is one); kLaSlowBytes long.
__host__ __device__ inline size_t la_slow_offset(int E, int H, size_t stride, int staged) {
  const size_t end = staged ? la_stage_offset(E, H) + la_stage_bytes(E, H, stride)
                            : 2 * (size_t)E * E * sizeof(float);
  return (end + 15) & ~size_t(15);
}

constexpr int kLaThreads = 128;
constexpr int kLaMaxCand = 65 * 32;  // (target + 64 substitutes) x 32 servers
constexpr int kLaTerms = 2048;       // (candidate, k') terms per pass

struct LaSmem {
  uint32_t code[kLaMaxCand];  // expert | server << 8 | substitute << 16
  float cost0[kLaMaxCand];    // A(a, s, m) + Cq: Eq. 43 without Phi
  float qn[kLaMaxCand];       // accumulated loss after this candidate (Eq. 44)
  float terms[kLaTerms];
  float U[32 * 64];           // H = 3, 4: Phi^(1)(m2, k2) with every budget check passing
  float qmax1[64];            // H = 3, 4: largest substitute loss Phi^(1)(., k2) can consider
  unsigned long long best;
  int n;
  int ns;                     // H = 3: pairs listed by phi_term2_split
};

__global__ void __launch_bounds__(kLaThreads) lookahead_select_kernel(
    const int32_t* __restrict__ topk_idx, int T, int E, int k, const uint8_t* __restrict__ tab,
    Lookahead la, const uint8_t* __restrict__ home, uint8_t* __restrict__ loc,
    float* __restrict__ qhat, int32_t* __restrict__ chosen_expert,
    uint8_t* __restrict__ chosen_server, uint8_t* __restrict__ kind_out,
    int32_t* __restrict__ counters) {
  pdl_trigger();  // launched with launch_pdl: no global access before pdl_wait
  pdl_wait();
  __shared__ SelSmem sm;
  __shared__ LaSmem cs;
  extern __shared__ __align__(16) float s_dyn[];
  float* s_Q = s_dyn;
  float* s_Cq = s_dyn + E * E;
  const int t = blockIdx.x;
  if (t >= T) return;
  if (!load_tables(tab, E, sm, s_Q, s_Cq)) return;
  // the next H - 1 layers' tables and transitions: read in place, or from a
  // shared-memory copy (every Phi term reads them along serial chains)
  const uint8_t* tn = tab + la.stride;
  const float* Pn = la.P;
  if (la.staged && la.H > 1) {
    uint8_t* st_tab = reinterpret_cast<uint8_t*>(s_dyn) + la_stage_offset(E, la.H);
    float* st_P = reinterpret_cast<float*>(st_tab + (size_t)(la.H - 1) * la.stride);
    const size_t tb = (size_t)(la.H - 1) * la.stride;  // a multiple of 16
    const size_t pn = (size_t)(la.H - 1) * E * E;
    if (((reinterpret_cast<uintptr_t>(tn) | reinterpret_cast<uintptr_t>(la.P)) & 15u) == 0) {
      const uint4* src = reinterpret_cast<const uint4*>(tn);
#pragma unroll 4
      for (size_t i = threadIdx.x; i < tb / 16; i += blockDim.x)
        reinterpret_cast<uint4*>(st_tab)[i] = __ldg(src + i);
    } else {
      const uint32_t* src = reinterpret_cast<const uint32_t*>(tn);
      for (size_t i = threadIdx.x; i < tb / 4; i += blockDim.x)
        reinterpret_cast<uint32_t*>(st_tab)[i] = src[i];
    }
    for (size_t i = threadIdx.x; i < pn; i += blockDim.x) st_P[i] = la.P[i];
    tn = st_tab;
    Pn = st_P;
  }
  __syncthreads();
  const int M = reinterpret_cast<const int32_t*>(tab)[2];
  const float qbar = reinterpret_cast<const float*>(tab)[5];
  const float* gA = reinterpret_cast<const float*>(tab + off_a(E));
  const int tid = threadIdx.x;
  const int a = home[t];
  const int s = (loc != nullptr) ? loc[t] : a;
  if (a >= M || s >= M) {
    if (tid == 0) report(&g_err_route, ORDERMOE_DEV_BAD_INDEX, t);
    return;
  }
  unsigned long long taken = 0;
  for (int j = 0; j < k; ++j) {
    const int r = topk_idx[(size_t)t * k + j];
    if (r < 0 || r >= E) return;  // -1: a token whose logits held a NaN (reported)
    taken |= 1ull << r;
  }
  const float* Aas = gA + ((size_t)a * M + s) * M;
  const int cpp = kLaTerms / E;  // candidates per pass
  float q = (qhat != nullptr) ? qhat[t] : 0.0f;
  const bool memo = (la.H == 3) && !(q < 0.0f);  // accumulated losses are never negative
  const bool memo4 = (la.H == 4) && !(q < 0.0f);
  float* U2 = s_dyn + 2 * E * E;  // H = 4: Phi^(2)(m2, k2) with every check passing, [32][E]
  float* qmax2 = U2 + 32 * E;     // H = 4: largest loss Phi^(2)(., k2) adds at its level
  float qmaxL1 = -INFINITY;       // H = 4: largest such loss one level deeper
  LaSlow slow{};                  // H = 3: the listed pairs
  if (memo) {
    uint8_t* sp = reinterpret_cast<uint8_t*>(s_dyn) + la_slow_offset(E, 3, la.stride, la.staged);
    slow.code = reinterpret_cast<uint32_t*>(sp);
    slow.base = reinterpret_cast<float*>(sp + (size_t)kLaSlow * 4);
    slow.q2 = slow.base + kLaSlow;
    slow.terms = slow.q2 + kLaSlow;
  }
  // the largest substitute loss lookahead_phi<1> on tables tl and transitions Pl
  // can add for expert kx (targets with P(kx -> k') != 0; -inf: none)
  auto qmax_of = [&](const uint8_t* tl, const float* Pl, int kx) {
    const float* Ql = reinterpret_cast<const float*>(tl + kOffQtab);
    const unsigned long long* sbl = reinterpret_cast<const unsigned long long*>(tl + kOffSubst);
    float mx = -INFINITY;
    for (int kt = 0; kt < E; ++kt) {
      if (ldt(Pl + (size_t)kx * E + kt) == 0.0f) continue;
      unsigned long long sb = ldt(sbl + kt);
      while (sb) {
        const int k3 = __ffsll(static_cast<long long>(sb)) - 1;
        sb &= sb - 1;
        mx = fmaxf(mx, ldt(Ql + kt * E + k3));
      }
    }
    return mx;
  };
  if (memo || memo4) {
    // the deepest level's tables (layer l + H - 1) and transitions into it
    const int dl = la.H - 1;
    const uint8_t* td = tn + (dl - 1) * la.stride;
    const float* Pd = Pn + (size_t)(dl - 1) * E * E;
    for (int k2 = tid; k2 < E; k2 += blockDim.x) cs.qmax1[k2] = qmax_of(td, Pd, k2);
    // U[m2][k2] = lookahead_phi<1>(m2, k2, q = 0): the E terms of every entry
    // (one per next target k') in parallel, then each entry's terms added in
    // ascending k', skipping P = 0, as lookahead_phi<1> adds them (the same
    // fp32 value; one thread per entry walked all its terms before)
    const int per = kLaTerms / E;  // entries per pass
    for (int base = 0; base < M * E; base += per) {
      const int ne = min(per, M * E - base);
      for (int i = tid; i < ne * E; i += blockDim.x) {
        const int c = base + i / E, kt = i - (i / E) * E;
        const int m2 = c / E, k2 = c - (c / E) * E;
        cs.terms[i] = phi_term<1>(td, la.stride, Pd, E, M, a, m2, k2, kt, 0.0f, qbar);
      }
      __syncthreads();
      for (int cl = tid; cl < ne; cl += blockDim.x) {
        const int c = base + cl, k2 = c - (c / E) * E;
        float phi = 0.0f;
        for (int kt = 0; kt < E; ++kt)
          if (ldt(Pd + (size_t)k2 * E + kt) != 0.0f) phi = __fadd_rn(phi, cs.terms[cl * E + kt]);
        cs.U[c] = phi;
      }
      __syncthreads();
    }
  }
  if (memo4) {
    // one level up (layer l + 2): Phi^(2) at q = 0, through the U table above
    const uint8_t* t2 = tn + la.stride;
    const float* P2 = Pn + (size_t)E * E;
    for (int k2 = tid; k2 < E; k2 += blockDim.x) qmax2[k2] = qmax_of(t2, P2, k2);
    for (int i = tid; i < M * E; i += blockDim.x) {
      const int m2 = i / E, k2 = i - (i / E) * E;
      U2[i] = lookahead_phi2_memo(t2, la.stride, P2, E, M, a, m2, k2, 0.0f, qbar, cs.U, cs.qmax1);
    }
    for (int k3 = 0; k3 < E; ++k3) qmaxL1 = fmaxf(qmaxL1, cs.qmax1[k3]);
    __syncthreads();
  }
  int first_server = s;
  for (int j = 0; j < k; ++j) {
    const int r = topk_idx[(size_t)t * k + j];
    if (tid == 0) {
      cs.n = 0;
      cs.best = ~0ull;
    }
    __syncthreads();
    // candidates: thread i takes the target (i = 0) or substitute i - 1
    const int nsub = sm.nsub[r];
    for (int ki = tid; ki <= nsub; ki += blockDim.x) {
      const int kk = (ki == 0) ? r : sm.sublist[r * 64 + ki - 1];
      const bool sub = (ki != 0);
      float cq = 0.0f, qn = q;
      bool ok = true;
      if (sub) {
        ok = !((taken >> kk) & 1ull) && (__fadd_rn(q, s_Q[r * E + kk]) <= qbar);
        if (ok) {
          cq = s_Cq[r * E + kk];
          qn = __fadd_rn(q, s_Q[r * E + kk]);
        }
      }
      uint32_t pm = ok ? sm.pmask[kk] : 0u;
      int slot = atomicAdd(&cs.n, __popc(pm));
      while (pm) {
        const int m = __ffs(pm) - 1;
        pm &= pm - 1;
        cs.code[slot] = static_cast<uint32_t>(kk) | (static_cast<uint32_t>(m) << 8) |
                        (sub ? (1u << 16) : 0u);
        cs.cost0[slot] = __fadd_rn(ldt(Aas + m), cq);
        cs.qn[slot] = qn;
        ++slot;
      }
    }
    __syncthreads();
    const int n = cs.n;
    for (int base = 0; base < n; base += cpp) {
      const int nc = min(cpp, n - base);
      if (memo) {
        // H = 3: each (candidate, k') item takes its pairs whose Phi^(1) is in
        // U and lists the others; the listed pairs' Phi^(1) is then evaluated
        // with its E terms in parallel and added in ascending k'' as
        // lookahead_phi<1> adds them, and each pair's cost joins its item's
        // minimum (a token near its budget has many such pairs, which one
        // thread used to walk one after another)
        if (tid == 0) cs.ns = 0;
        __syncthreads();
        uint32_t* key = reinterpret_cast<uint32_t*>(cs.terms);
        for (int i = tid; i < nc * E; i += blockDim.x) {
          const int c = base + i / E, kt = i - (i / E) * E;
          const uint32_t code = cs.code[c];
          const int cm = static_cast<int>((code >> 8) & 0xFFu), ck = static_cast<int>(code & 0xFFu);
          if (ldt(Pn + (size_t)ck * E + kt) != 0.0f)
            key[i] = phi_term2_split(tn, la.stride, Pn, E, M, a, cm, ck, kt, cs.qn[c], qbar, cs.U,
                                     cs.qmax1, i, slow, &cs.ns);
        }
        __syncthreads();
        const int ns = min(cs.ns, kLaSlow);
        const int per2 = kLaSlowTerms / E;
        for (int sb = 0; sb < ns; sb += per2) {
          const int ne = min(per2, ns - sb);
          for (int j = tid; j < ne * E; j += blockDim.x) {
            const int e = sb + j / E, k3 = j - (j / E) * E;
            const uint32_t sc = slow.code[e];
            slow.terms[j] = phi_term<1>(tn + la.stride, la.stride, Pn + E * E, E, M, a,
                                        static_cast<int>((sc >> 8) & 0xFFu),
                                        static_cast<int>(sc & 0xFFu), k3, slow.q2[e], qbar);
          }
          __syncthreads();
          for (int el = tid; el < ne; el += blockDim.x) {
            const uint32_t sc = slow.code[sb + el];
            const int kk = static_cast<int>(sc & 0xFFu);
            const float* P2 = Pn + (size_t)E * E + (size_t)kk * E;
            float phi1 = 0.0f;
            for (int k3 = 0; k3 < E; ++k3)
              if (ldt(P2 + k3) != 0.0f) phi1 = __fadd_rn(phi1, slow.terms[el * E + k3]);
            atomicMin(&key[sc >> 16], min_key(__fadd_rn(slow.base[sb + el], phi1)));
          }
          __syncthreads();
        }
      } else {
        for (int i = tid; i < nc * E; i += blockDim.x) {
          const int c = base + i / E, kt = i - (i / E) * E;
          const uint32_t code = cs.code[c];
          const int cm = static_cast<int>((code >> 8) & 0xFFu), ck = static_cast<int>(code & 0xFFu);
          cs.terms[i] = memo4 ? phi_term3_memo(tn, la.stride, Pn, E, M, a, cm, ck, kt, cs.qn[c],
                                               qbar, U2, qmax2, qmaxL1, cs.U, cs.qmax1)
                              : phi_term_h(la.H, tn, la.stride, Pn, E, M, a, cm, ck, kt, cs.qn[c],
                                           qbar);
        }
        __syncthreads();
      }
      for (int cl = tid; cl < nc; cl += blockDim.x) {
        const uint32_t code = cs.code[base + cl];
        const int kk = static_cast<int>(code & 0xFFu), m = static_cast<int>((code >> 8) & 0xFFu);
        const unsigned sub = (code >> 16) & 1u;
        float phi = 0.0f;
        for (int kt = 0; kt < E; ++kt) {
          const float p = ldt(Pn + (size_t)kk * E + kt);
          if (p == 0.0f) continue;
          const float term = cs.terms[cl * E + kt];
          phi = __fadd_rn(phi, memo ? __fmul_rn(p, from_min_key(__float_as_uint(term))) : term);
        }
        const float cost = __fadd_rn(cs.cost0[base + cl], phi);
        const unsigned long long key =
            (static_cast<unsigned long long>(__float_as_uint(cost)) << 32) |
            (static_cast<unsigned long long>(sub) << 31) |
            (static_cast<unsigned long long>(m != s ? 1u : 0u) << 30) |
            (static_cast<unsigned long long>(m) << 8) | static_cast<unsigned long long>(kk);
        atomicMin(&cs.best, key);
      }
      __syncthreads();
    }
    const unsigned long long best = cs.best;
    int kstar, mstar, kd;
    if (best == ~0ull) {
      if (tid == 0) report(&g_err_route, ORDERMOE_DEV_NO_CANDIDATE, t);
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
    if (tid == 0) {
      chosen_expert[(size_t)t * k + j] = kstar;
      chosen_server[(size_t)t * k + j] = static_cast<uint8_t>(mstar);
      kind_out[(size_t)t * k + j] = static_cast<uint8_t>(kd);
      if (counters != nullptr) atomicAdd(&counters[kd], 1);
    }
    __syncthreads();  // the candidate arrays are rewritten for the next slot
  }
  if (tid == 0 && loc != nullptr) {
    loc[t] = static_cast<uint8_t>(first_server);
    qhat[t] = q;
  }
}

// ---------------------------------------------------------------------------
// Router on tcgen05 + selection. A cluster of S CTAs (S = 1..8) handles 128
// tokens: CTA r of the cluster accumulates logits = X W_r^T over its share of
// the K blocks (M = 128 tokens, N = NE >= E padded to 16/32/64) in TMEM. Its
// epilogue thread i of warp w (w = 2..5) reads TMEM lane 32 (w % 4) + i (token
// 32 (w % 4) + i); ranks > 0 store their partial logits into rank 0's shared
// memory (distributed shared memory), and after a cluster barrier rank 0 adds
// the partials in rank order (deterministic) and runs select_token. Splitting
// K lets a few hundred tokens (decode) still stream X over many SMs. The
// partials are laid out [rank - 1][NE / 4][128 tokens][4], so that the 32
// tokens of a warp store and load 16-byte vectors at consecutive addresses
// (no bank conflicts). While the TMA and MMA warps run, rank 0's epilogue
// warps load the selection tables (the delay table too, when small) and
// each token's home, location and loss.
// Warp 0 issues the TMA loads (X: 128 x 64 box; W_r: NE x 64 box, rows >= E
// zero-filled), warp 1 the MMAs; mbarrier ring; bounded waits.
namespace rt {
constexpr int BK = 64;
constexpr int A_BYTES = 128 * BK * 2;
constexpr int THREADS = 192;
// Only layers of up to 16 experts (NE = 16) select inside the router; for
// more experts it writes the targets and a selection kernel selects, so the
// wider instantiations keep no tables and give that space to the X ring.
template <int NE>
constexpr bool selects() { return NE <= 16; }
// stages of (16 KB + NE x 128 B) in flight per CTA, and the largest cluster,
// sized so the ring, the partial logits of ranks 1..S-1 and (NE = 16) the
// tables and the staged delay table fit in 227 KB beside the static
// selection tables
template <int NE>
constexpr int stages() { return NE <= 16 ? 8 : (NE <= 32 ? 8 : 7); }
template <int NE>
constexpr int max_split() { return NE <= 16 ? 8 : (NE <= 32 ? 4 : 2); }
template <int NE>
constexpr int smem_bytes(int E) {
  return 1024 + stages<NE>() * (A_BYTES + NE * BK * 2) + 256 +
         (max_split<NE>() - 1) * 128 * NE * 4 + (selects<NE>() ? 8 * E * E + 4 * kDelayStage : 0);
}
static_assert(smem_bytes<16>(16) + sizeof(SelSmem) <= 227 * 1024, "router shared memory");
static_assert(smem_bytes<32>(32) + sizeof(SelSmem) <= 227 * 1024, "router shared memory");
static_assert(smem_bytes<64>(64) + sizeof(SelSmem) <= 227 * 1024, "router shared memory");
}  // namespace rt

template <int NE>
struct RouterSmem {
  uint64_t full[rt::stages<NE>()];
  uint64_t empty[rt::stages<NE>()];
  uint64_t tfull;
  uint64_t drain;
  uint32_t tmem_base;
  int abort;
  int zero;
};

template <int NE>
__global__ void __launch_bounds__(rt::THREADS, 1) router_select_kernel(
    const __grid_constant__ CUtensorMap mapX, const __grid_constant__ CUtensorMap mapW, int T,
    int E, int d, int k, int renorm, const uint8_t* __restrict__ tab,
    const uint8_t* __restrict__ home, uint8_t* __restrict__ loc, float* __restrict__ qhat,
    float* __restrict__ logits_out, int32_t* __restrict__ topk_idx, float* __restrict__ topk_w,
    int32_t* __restrict__ chosen_expert, uint8_t* __restrict__ chosen_server,
    uint8_t* __restrict__ kind_out, int32_t* __restrict__ counters, uint64_t limit_ns, int split,
    Lookahead la) {
  pdl_trigger();  // launched with launch_pdl: shared memory, barrier and TMEM set-up first
  constexpr int B_BYTES = NE * rt::BK * 2;
  constexpr int STAGE_BYTES = rt::A_BYTES + B_BYTES;
  constexpr int STAGES = rt::stages<NE>();
  constexpr int TMEM_COLS = NE <= 32 ? 32 : NE;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* tiles = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  RouterSmem<NE>& s = *reinterpret_cast<RouterSmem<NE>*>(tiles + STAGES * STAGE_BYTES);
  // partials of ranks 1..split-1: [split - 1][NE / 4][128][4]
  float* red = reinterpret_cast<float*>(tiles + STAGES * STAGE_BYTES + 256);
  float* s_Q = red + (rt::max_split<NE>() - 1) * 128 * NE;
  float* s_Cq = s_Q + E * E;
  float* s_A = s_Cq + E * E;
  __shared__ SelSmem sm;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t rank = split > 1 ? cluster_ctarank() : 0;
  const int tile = blockIdx.x / split;
  const int m0 = tile * 128;
  const int kblocks_all = d / rt::BK;
  const int per = (kblocks_all + split - 1) / split;
  const int kb_begin = static_cast<int>(rank) * per;
  const int kb_end = min(kblocks_all, kb_begin + per);
  const int kblocks = kb_end > kb_begin ? kb_end - kb_begin : 0;

  if (tid == 0) {
    for (int i = 0; i < STAGES; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.empty[i], 1);
    }
    mbar_init(&s.tfull, 1);
    mbar_init(&s.drain, 1);
    s.abort = 0;
    s.zero = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_map(&mapX);
    tma_prefetch_map(&mapW);
  }
  if (warp == 1) {
    tmem_alloc(&s.tmem_base, TMEM_COLS);
    tmem_relinquish();
  }
  bool tables_ok = true;  // rank 0's epilogue warps load the tables during the main loop
  const float* Atab = nullptr;
  int pre_a = 0, pre_s = 0;  // the token's home and location, loaded during the main loop
  float pre_q = 0.0f;
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait();  // the previous kernel's outputs (X, tables, state) are ready
  const uint32_t tmem_base = s.tmem_base;
  volatile int* abort = &s.abort;
  uint32_t issued_mask = 0, last_phase_bits = 0;
  bool mma_issued = false;
  float lg[NE];
  int kind_count[4] = {0, 0, 0, 0};

  if (warp == 0) {
    if (lane == 0) {
      for (int i = 0; i < kblocks && !*abort; ++i) {
        const int stage = i % STAGES;
        const uint32_t phase = (i / STAGES) & 1;
        if (!mbar_wait(&s.empty[stage], phase ^ 1u, limit_ns, abort)) {
          if (!*abort) report(&g_err_route, ORDERMOE_DEV_WAIT_TIMEOUT, 21);
          *abort = 1;
          break;
        }
        uint8_t* sa = tiles + stage * STAGE_BYTES;
        const int kb = kb_begin + i;
        mbar_arrive_expect_tx(&s.full[stage], STAGE_BYTES);
        tma_load_2d(sa, &mapX, &s.full[stage], kb * rt::BK, m0);
        tma_load_2d(sa + rt::A_BYTES, &mapW, &s.full[stage], kb * rt::BK, 0);
        issued_mask |= 1u << stage;
        last_phase_bits = (last_phase_bits & ~(1u << stage)) | (phase << stage);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t IDESC = idesc_bf16_f32(128, NE);
      bool ok = true;
      for (int i = 0; i < kblocks && !*abort; ++i) {
        const int stage = i % STAGES;
        const uint32_t phase = (i / STAGES) & 1;
        if (!mbar_wait(&s.full[stage], phase, limit_ns, abort)) {
          if (!*abort) report(&g_err_route, ORDERMOE_DEV_WAIT_TIMEOUT, 22);
          *abort = 1;
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t a0 = smem_u32(tiles + stage * STAGE_BYTES);
        const uint32_t b0 = a0 + rt::A_BYTES;
#pragma unroll
        for (int kk = 0; kk < rt::BK / 16; ++kk)
          mma_bf16(tmem_base, sdesc_kmajor_sw128(a0 + kk * 32), sdesc_kmajor_sw128(b0 + kk * 32),
                   IDESC, (i | kk) != 0 ? 1u : 0u);
        mma_issued = true;
        mma_commit(&s.empty[stage]);
      }
      if (ok && !*abort) {
        if (mma_issued) mma_commit(&s.tfull);
        else mbar_arrive(&s.tfull);  // empty K share: nothing to wait for
      }
    }
  } else {
    // the selection tables, while the TMA and MMA warps run (named barrier 1:
    // the 128 epilogue threads)
    if (rank == 0) {
      if (!rt::selects<NE>() || la.H > 1 || la.topk_only) {  // targets only: a selection kernel reads the tables
        if (tid - 64 < 4) sm.kind[tid - 64] = 0;
      } else {
        const int t = m0 + (warp & 3) * 32 + lane;
        if (t < T) {
          pre_a = home[t];
          pre_s = (loc != nullptr) ? loc[t] : pre_a;  // no state given: first layer (Eq. 36)
          pre_q = (qhat != nullptr) ? qhat[t] : 0.0f;
        }
        tables_ok = load_tables_range(tab, E, sm, s_Q, s_Cq, tid - 64, 128);
        Atab = load_delay_range(tab, E, s_A, tid - 64, 128);
      }
    }
    asm volatile("bar.sync 1, 128;" ::: "memory");
    // epilogue part 1: this CTA's partial logits
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const bool ok = __all_sync(0xffffffffu, mbar_wait(&s.tfull, 0, limit_ns, abort));
    if (!ok) {
      if (lane == 0 && !*abort) report(&g_err_route, ORDERMOE_DEV_WAIT_TIMEOUT, 23);
      *abort = 1;
    } else {
      tc_fence_after();
#pragma unroll
      for (int c = 0; c < NE; c += 32) {
        uint32_t v[32];
        tmem_ld32(tmem_base + (static_cast<uint32_t>(q * 32) << 16) + c, v);
        tmem_ld_wait();
#pragma unroll
        for (int i = 0; i < 32; ++i)
          if (c + i < NE) lg[c + i] = kblocks > 0 ? __uint_as_float(v[i]) : 0.0f;
      }
      tc_fence_before();
      if (rank > 0) {
        // partial logits of this rank -> red[rank - 1][c / 4][row][c % 4] in rank 0's
        // shared memory
        const uint32_t dst =
            mapa_shared(smem_u32(red + ((size_t)(rank - 1) * (NE / 4) * 128 + row) * 4), 0);
#pragma unroll
        for (int c = 0; c < NE; c += 4)
          asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(dst + c * 128 * 4),
                       "f"(lg[c]), "f"(lg[c + 1]), "f"(lg[c + 2]), "f"(lg[c + 3])
                       : "memory");
      }
    }
  }
  if (split > 1) cluster_sync();  // partials visible in rank 0
  if (warp >= 2 && rank == 0 && !*abort) {
    // epilogue part 2: full logits (partials in rank order) and the selection
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const int t = m0 + row;
    for (int r = 1; r < split; ++r) {
      const float4* src = reinterpret_cast<const float4*>(red) + (size_t)(r - 1) * (NE / 4) * 128 + row;
#pragma unroll
      for (int c = 0; c < NE; c += 4) {
        const float4 p = src[(c / 4) * 128];
        lg[c] += p.x;
        lg[c + 1] += p.y;
        lg[c + 2] += p.z;
        lg[c + 3] += p.w;
      }
    }
#pragma unroll
    for (int e = 0; e < NE; ++e)  // padding past E for select_token
      if (e >= E) lg[e] = -INFINITY;
    if (t < T && tables_ok) {
      if (logits_out != nullptr) {
#pragma unroll
        for (int e = 0; e < NE; ++e)  // constant indices keep lg[] in registers
          if (e < E) logits_out[(size_t)t * E + e] = lg[e];
      }
      // the token's logits into this thread's column of partial slot 0 (read above)
      float4* col = reinterpret_cast<float4*>(red) + row;
#pragma unroll
      for (int c = 0; c < NE; c += 4)
        col[(c / 4) * 128] = make_float4(lg[c], lg[c + 1], lg[c + 2], lg[c + 3]);
      const int M = reinterpret_cast<const int32_t*>(tab)[2];
      const float qbar = reinterpret_cast<const float*>(tab)[5];
      select_token(t, ColLogits{col}, E, k, renorm, M, qbar, Atab, tab, la, sm, s_Q, s_Cq, pre_a,
                   pre_s, pre_q, loc, qhat, topk_idx, topk_w, chosen_expert, chosen_server,
                   kind_out, kind_count, !rt::selects<NE>() || la.H > 1 || la.topk_only);
    }
    flush_kind_counts(sm, kind_count, counters);
  }

  __syncthreads();
  if (s.abort) {
    volatile int* never = &s.zero;
    if (warp == 0 && lane == 0)
      for (int st = 0; st < STAGES; ++st)
        if ((issued_mask >> st) & 1u) mbar_wait(&s.full[st], (last_phase_bits >> st) & 1u, limit_ns, never);
    if (warp == 1 && lane == 0 && mma_issued) {
      mma_commit(&s.drain);
      mbar_wait(&s.drain, 0, limit_ns, never);
    }
    __syncthreads();
  }
  if (rank == 0 && counters != nullptr && tid < 4 && sm.kind[tid]) atomicAdd(&counters[tid], sm.kind[tid]);
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, TMEM_COLS);
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
  OM_TRACE();
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

static int launch_lookahead_select(const int32_t* topk_idx, int T, int E, int k,
                                   const uint8_t* tb, Lookahead la, const uint8_t* home,
                                   uint8_t* loc, float* qhat, int32_t* chosen_expert,
                                   uint8_t* chosen_server, uint8_t* kind, int32_t* counters,
                                   size_t tab_smem, cudaStream_t stream) {
  if (T <= 0) return ORDERMOE_OK;
  if (la.H == 4) tab_smem += sizeof(float) * (32 * E + E);  // the Phi^(2) table and its bounds
  // the next layers' tables and transitions in shared memory when they fit
  la.staged = 0;
  if (la.H > 1) {
    const size_t staged = la_stage_offset(E, la.H) + la_stage_bytes(E, la.H, la.stride);
    if (staged <= 160 * 1024) {
      tab_smem = staged;
      la.staged = 1;
    }
  }
  if (la.H == 3) tab_smem = la_slow_offset(E, 3, la.stride, la.staged) + kLaSlowBytes;
  cudaFuncSetAttribute(lookahead_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)tab_smem);
  OM_LAUNCH_PDL("lookahead_select_kernel", lookahead_select_kernel, dim3(T), dim3(kLaThreads),
                tab_smem, stream, topk_idx, T, E, k, tb, la, home, loc, qhat, chosen_expert,
                chosen_server, kind, counters);
  return ORDERMOE_OK;
}

static int launch_select_lanes(const int32_t* topk_idx, int T, int E, int k, const uint8_t* tb,
                               const uint8_t* home, uint8_t* loc, float* qhat,
                               int32_t* chosen_expert, uint8_t* chosen_server, uint8_t* kind,
                               int32_t* counters, size_t tab_smem, cudaStream_t stream) {
  if (T <= 0) return ORDERMOE_OK;
  const int per_block = (kLaneThreads / 32) * kLaneTokens;
  long long blocks = (T + per_block - 1) / per_block;
  const long long cap = 4LL * num_sms();
  if (blocks > cap) blocks = cap;
  cudaFuncSetAttribute(select_lanes_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       (int)tab_smem);
  OM_LAUNCH_PDL("select_lanes_kernel", select_lanes_kernel, dim3(static_cast<int>(blocks)),
                dim3(kLaneThreads), tab_smem, stream, topk_idx, T, E, k, tb, home, loc, qhat,
                chosen_expert, chosen_server, kind, counters);
  return ORDERMOE_OK;
}

static int route_select_impl(const uint16_t* X, const uint16_t* W_r, const float* logits_in, int T,
                             int E, int d, int k, int renorm, const void* tables,
                             size_t tables_bytes_, Lookahead la, const uint8_t* home, uint8_t* loc,
                             float* qhat, float* logits_out, int32_t* topk_idx, float* topk_w,
                             int32_t* chosen_expert, uint8_t* chosen_server, uint8_t* kind,
                             int32_t* counters, cudaStream_t stream) {
  if (T < 0) return fail(ORDERMOE_ERR_INVALID_ARG, "route_select: T < 0");
  if (E <= 0 || E > ORDERMOE_MAX_EXPERTS || k <= 0 || k > ORDERMOE_MAX_TOPK || k > E)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "route_select: need 1 <= k <= min(E, 8), E <= 64");
  if (!tables || !home || !topk_idx || !topk_w || !chosen_expert || !chosen_server || !kind)
    return fail(ORDERMOE_ERR_INVALID_ARG, "route_select: null pointer");
  if ((loc == nullptr) != (qhat == nullptr))
    return fail(ORDERMOE_ERR_INVALID_ARG, "route_select: give both loc and qhat, or neither");
  if (logits_in == nullptr) {
    if (!X || !W_r) return fail(ORDERMOE_ERR_INVALID_ARG, "route_select: X/W_r null without logits_in");
    if (d <= 0 || d % 64 != 0)
      return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "route_select: d must be a positive multiple of 64");
    if (!aligned16(X) || !aligned16(W_r))
      return fail(ORDERMOE_ERR_INVALID_ARG, "route_select: X and W_r must be 16-byte aligned");
  }
  if (tables_bytes_ < om::tables_bytes(E, 1))
    return fail(ORDERMOE_ERR_INVALID_ARG, "route_select: tables buffer smaller than E needs");
  if (T == 0) return ORDERMOE_OK;
  const uint8_t* tb = static_cast<const uint8_t*>(tables);
  const size_t tab_smem = sizeof(float) * 2 * E * E;  // the look-ahead and lane kernels'
  const size_t sel_smem = tab_smem + sizeof(float) * kDelayStage;  // + the staged delay table
  const int blocks = (T + 127) / 128;
  if (logits_in != nullptr) {
    cudaError_t sel_err = cudaSuccess;
#define OM_SEL_LAUNCH(EM)                                                                        \
  do {                                                                                           \
    const size_t lg_smem = sel_smem + sizeof(float) * EM * 128; /* + the logits' chunks */      \
    cudaFuncSetAttribute(select_kernel<EM>, cudaFuncAttributeMaxDynamicSharedMemorySize,         \
                         (int)lg_smem);                                                          \
    sel_err = launch_pdl(select_kernel<EM>, dim3(blocks), dim3(128), lg_smem, stream,            \
                         logits_in, T, E, k, renorm, tb, home, loc, qhat, logits_out, topk_idx,   \
                         topk_w, chosen_expert, chosen_server, kind, counters, la);              \
  } while (0)
    if (E <= 8) OM_SEL_LAUNCH(8);
    else if (E <= 16) OM_SEL_LAUNCH(16);
    else if (E <= 32) OM_SEL_LAUNCH(32);
    else OM_SEL_LAUNCH(64);
#undef OM_SEL_LAUNCH
    if (sel_err != cudaSuccess) return cuda_fail(sel_err, "select_kernel");
    return la.H > 1 ? launch_lookahead_select(topk_idx, T, E, k, tb, la, home, loc, qhat,
                                              chosen_expert, chosen_server, kind, counters,
                                              tab_smem, stream)
                    : ORDERMOE_OK;
  }
  // many experts (long candidate lists per slot): the router writes the
  // targets and select_lanes_kernel selects with eight lanes per token
  const bool lanes = la.H == 1 && E > 16;
  if (lanes) la.topk_only = 1;
  CUtensorMap mX, mW;
  int rc;
  const int NE = E <= 16 ? 16 : (E <= 32 ? 32 : 64);
  if ((rc = make_tmap_bf16(&mX, X, T, d, 128))) return rc;
  if ((rc = make_tmap_bf16(&mW, W_r, E, d, NE))) return rc;
  const uint64_t lim = wait_limit_ns();
  // split K over a cluster so that about one CTA per SM streams X
  const int kblocks = d / rt::BK;
  const int smax = NE == 16 ? rt::max_split<16>() : (NE == 32 ? rt::max_split<32>() : rt::max_split<64>());
  int split = 1;
  while (split * 2 <= smax && (long long)blocks * split * 2 <= num_sms() && split * 2 <= kblocks)
    split *= 2;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(blocks * split, 1, 1);
  cfg.blockDim = dim3(rt::THREADS, 1, 1);
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = split;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;  // waits in the kernel
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_on(stream) ? 2 : 1;
  cudaError_t le;
#define OM_RT_LAUNCH(N)                                                                          \
  do {                                                                                           \
    cfg.dynamicSmemBytes = rt::smem_bytes<N>(E);                                                 \
    cudaFuncSetAttribute(router_select_kernel<N>, cudaFuncAttributeMaxDynamicSharedMemorySize,   \
                         (int)cfg.dynamicSmemBytes);                                             \
    le = cudaLaunchKernelEx(&cfg, router_select_kernel<N>, mX, mW, T, E, d, k, renorm, tb, home, \
                            loc, qhat, logits_out, topk_idx, topk_w, chosen_expert,              \
                            chosen_server, kind, counters, lim, split, la);                      \
  } while (0)
  if (NE == 16) OM_RT_LAUNCH(16);
  else if (NE == 32) OM_RT_LAUNCH(32);
  else OM_RT_LAUNCH(64);
#undef OM_RT_LAUNCH
  if (le != cudaSuccess) return cuda_fail(le, "router_select_kernel launch");
  OM_LAUNCHED("router_select_kernel");
  if (la.H > 1)
    return launch_lookahead_select(topk_idx, T, E, k, tb, la, home, loc, qhat, chosen_expert,
                                   chosen_server, kind, counters, tab_smem, stream);
  if (lanes)
    return launch_select_lanes(topk_idx, T, E, k, tb, home, loc, qhat, chosen_expert,
                               chosen_server, kind, counters, tab_smem, stream);
  return ORDERMOE_OK;
}

extern "C" int ordermoe_route_select(const uint16_t* X, const uint16_t* W_r, const float* logits_in,
                                     int T, int E, int d, int k, int renorm, const void* tables,
                                     size_t tables_bytes_, const uint8_t* home, uint8_t* loc,
                                     float* qhat, float* logits_out, int32_t* topk_idx,
                                     float* topk_w, int32_t* chosen_expert,
                                     uint8_t* chosen_server, uint8_t* kind, int32_t* counters,
                                     ordermoe_stream_t stream) {
  OM_TRACE();
  Lookahead la{1, 0, nullptr};
  return route_select_impl(X, W_r, logits_in, T, E, d, k, renorm, tables, tables_bytes_, la, home,
                           loc, qhat, logits_out, topk_idx, topk_w, chosen_expert, chosen_server,
                           kind, counters, stream);
}

extern "C" int ordermoe_route_select_lookahead(
    const uint16_t* X, const uint16_t* W_r, const float* logits_in, int T, int E, int d, int k,
    int renorm, const void* tables, size_t tables_stride, int H, const float* P,
    const uint8_t* home, uint8_t* loc, float* qhat, float* logits_out, int32_t* topk_idx,
    float* topk_w, int32_t* chosen_expert, uint8_t* chosen_server, uint8_t* kind,
    int32_t* counters, ordermoe_stream_t stream) {
  OM_TRACE();
  if (H < 1 || H > 4) return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "route_select_lookahead: need 1 <= H <= 4");
  if (E <= 0 || E > ORDERMOE_MAX_EXPERTS)
    return fail(ORDERMOE_ERR_UNSUPPORTED_SHAPE, "route_select_lookahead: need 1 <= E <= 64");
  if (H > 1 && (!P || tables_stride < om::tables_bytes(E, 1) || (tables_stride & 15u)))
    return fail(ORDERMOE_ERR_INVALID_ARG,
                "route_select_lookahead: need P and a 16-byte multiple table stride for H > 1");
  Lookahead la{H, tables_stride, P};
  return route_select_impl(X, W_r, logits_in, T, E, d, k, renorm, tables, tables_stride, la, home,
                           loc, qhat, logits_out, topk_idx, topk_w, chosen_expert, chosen_server,
                           kind, counters, stream);
}
