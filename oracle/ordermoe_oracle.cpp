// OrderMoE CPU oracle.
//
// TEST INFRASTRUCTURE ONLY. This file is the slow, plain reference that the
// CUDA library is checked against. Only the test suite, the smoke check in
// __graft_entry__.py and the CPU-baseline leg of bench.py may load it. It
// shares no code, header, table or helper with the CUDA library, and the CUDA
// library never calls it.
//
// Paper: "OrderMoE: an expert similarity driven distributed edge MoE
// inference" (arXiv 2607.17154). Every function names the section and
// equation it follows. Floating point is fp64 unless a step is stated to run
// in fp32 (the selection's cost compares, which the method decides in fp32
// on both sides from identical fp32 tables). Build with -ffp-contract=off so
// that no multiply-add is fused.
//
// Readings where the paper is silent or garbled:
//  * top-k > 1: the selection of Alg. 2 runs once per routed slot, in rank
//    order; a substitute may not be an expert the token already routes to or
//    has already been given (every token keeps k distinct experts).
//  * the token location after a layer is the server of slot 0 (highest gate).
//  * phi in Eq. 18 is the identity.
//  * d_ref in Eq. 38 is the compute-only delay c/F_a on the home server a.
//  * argmin ties in Eq. 43: lower cost, then exact before substitute, then
//    the token's current server, then lower server id, then lower expert id.
//  * grouping (Eqs. 24-25): experts in decreasing frequency (ties: lower
//    index); argmax ties go to the earlier-created dominant; group id = the
//    dominant's creation order.
//  * placement (Eqs. 29-31): the within-layer order is memory demand desc,
//    then importance desc, then index asc; score ties go to the lower server;
//    the used memory b_m accumulates over layers (Alg. 1 initialises it once).
//  * redundancy (Eqs. 32-35): a replica's benefit is pi_m I (1 - y) / p; the
//    greedy takes the largest fitting benefit (ties: lower layer, server,
//    expert); pi_m is the share of tokens whose trajectory reaches server m.
#include <algorithm>
#include <cmath>
#include <limits>
#include <cstdint>
#include <cstring>
#include <vector>

#include <omp.h>

namespace {

float bf16_bits_to_float(uint16_t h) {
  uint32_t u = static_cast<uint32_t>(h) << 16;
  float f;
  std::memcpy(&f, &u, sizeof f);
  return f;
}

// Round-to-nearest-even fp32 -> bf16 (the rounding the bf16 format defines).
uint16_t float_to_bf16_bits(float f) {
  uint32_t u;
  std::memcpy(&u, &f, sizeof u);
  if ((u & 0x7fffffffu) > 0x7f800000u) return static_cast<uint16_t>((u >> 16) | 0x0040u);
  uint32_t lsb = (u >> 16) & 1u;
  u += 0x7fffu + lsb;
  return static_cast<uint16_t>(u >> 16);
}

double bf(const uint16_t* p, int64_t i) { return static_cast<double>(bf16_bits_to_float(p[i])); }

// Rank order used for top-k: larger logit first, equal logits by lower index.
bool ranks_before(float a, int ia, float b, int ib) {
  if (a != b) return a > b;
  return ia < ib;
}

}  // namespace

extern "C" {

// Status codes of this oracle (independent of the library's).
enum { ORC_OK = 0, ORC_BAD_ARG = 1, ORC_NAN = 2, ORC_CAPACITY = 3 };

// ---------------------------------------------------------------------------
// Router logits, Eq. 3 written per token: logits[t][e] = sum_c X[t][c] W[e][c]
// (the router's response; Alg. 2 obtains the target expert from it). fp64
// accumulation, stored as fp32.
int orc_router_logits(const uint16_t* X, const uint16_t* W, int T, int E, int d, float* logits) {
  if (T < 0 || E <= 0 || d <= 0) return ORC_BAD_ARG;
  for (int t = 0; t < T; ++t)
    for (int e = 0; e < E; ++e) {
      double acc = 0.0;
      for (int c = 0; c < d; ++c) acc += bf(X, (int64_t)t * d + c) * bf(W, (int64_t)e * d + c);
      logits[(int64_t)t * E + e] = static_cast<float>(acc);
    }
  return ORC_OK;
}

// Softmax over all E experts in fp64, then the k highest logits (ties: lower
// index). Gate weight of slot j = p[idx_j], renormalised over the k slots when
// renorm != 0. A NaN logit is an error.
int orc_topk(const float* logits, int T, int E, int k, int renorm, int32_t* idx, float* w) {
  if (T < 0 || E <= 0 || k <= 0 || k > E) return ORC_BAD_ARG;
  std::vector<int> order(E);
  std::vector<double> p(E);
  for (int t = 0; t < T; ++t) {
    const float* l = logits + (int64_t)t * E;
    for (int e = 0; e < E; ++e)
      if (std::isnan(l[e])) return ORC_NAN;
    for (int e = 0; e < E; ++e) order[e] = e;
    std::sort(order.begin(), order.end(),
              [&](int a, int b) { return ranks_before(l[a], a, l[b], b); });
    double mx = static_cast<double>(l[order[0]]);
    double s = 0.0;
    for (int e = 0; e < E; ++e) {
      p[e] = std::exp(static_cast<double>(l[e]) - mx);
      s += p[e];
    }
    for (int e = 0; e < E; ++e) p[e] /= s;
    double ssel = 0.0;
    for (int j = 0; j < k; ++j) ssel += p[order[j]];
    for (int j = 0; j < k; ++j) {
      idx[(int64_t)t * k + j] = order[j];
      double wj = renorm ? p[order[j]] / ssel : p[order[j]];
      w[(int64_t)t * k + j] = static_cast<float>(wj);
    }
  }
  return ORC_OK;
}

// ---------------------------------------------------------------------------
// Per-layer selection tables.
//   Qtab[r][k] = Q_l(r,k) of Eq. 18 with phi = identity, in fp32:
//                0 for k == r, else 0.5f * (1 - min(Sim,1)).
//   Cq[r][k]   = omega_Q * Q_l(r,k) / Qbar (the quality term of Eq. 38),
//                fp64 then rounded to fp32; 0 where Q_l = 0.
//   subst[r]   = bit set of R_{l,r} (Eq. 7): k != r in r's group with
//                Sim(r,k) >= theta.
//   A[a][s][m] = omega_T * d(s,m) / d_ref(a) (the delay term of Eq. 38) with
//                d(s,m) = 1(s != m)(z / B_{s,m} + tau_{s,m}) + c / F_m (Eq. 37)
//                and d_ref(a) = c / F_a; fp64 then rounded to fp32.
//   pmask[e]   = bit set of servers m with x_{m,e} = 1.
int orc_tables(const float* sim, const int32_t* group, const uint8_t* placement, int E, int M,
               float theta, float qbar, const double* F, const double* B, const double* tau,
               double z, double c, double omega_T, double omega_Q, float* Qtab, float* Cq,
               uint64_t* subst, float* A, uint32_t* pmask) {
  if (E <= 0 || E > 64 || M <= 0 || M > 32 || !(qbar >= 0.0f)) return ORC_BAD_ARG;
  for (int r = 0; r < E; ++r) {
    uint64_t bits = 0;
    for (int k = 0; k < E; ++k) {
      float s = sim[r * E + k];
      float q = 0.0f;
      if (k != r) q = 0.5f * (1.0f - std::min(s, 1.0f));
      Qtab[r * E + k] = q;
      float cq = 0.0f;
      if (q != 0.0f) cq = static_cast<float>(omega_Q * static_cast<double>(q) / static_cast<double>(qbar));
      Cq[r * E + k] = cq;
      if (k != r && group[k] == group[r] && s >= theta) bits |= (uint64_t)1 << k;
    }
    subst[r] = bits;
  }
  for (int a = 0; a < M; ++a) {
    double dref = c / F[a];
    for (int s = 0; s < M; ++s)
      for (int m = 0; m < M; ++m) {
        double comp = c / F[m];
        double dl = comp;
        if (s != m) {
          double trans = z / B[s * M + m] + tau[s * M + m];
          dl = trans + comp;
        }
        double num = omega_T * dl;
        A[((int64_t)a * M + s) * M + m] = static_cast<float>(num / dref);
      }
  }
  for (int e = 0; e < E; ++e) {
    uint32_t bits = 0;
    for (int m = 0; m < M; ++m)
      if (placement[m * E + e]) bits |= 1u << m;
    pmask[e] = bits;
  }
  return ORC_OK;
}

// ---------------------------------------------------------------------------
// Online server-expert selection, Alg. 2 with horizon H = 1 (Phi = 0,
// Section V-C), one routed slot at a time in rank order.
//   s = loc[t] (Eq. 36: the home server a(i) before the first layer),
//   feasible set (Eq. 40): (m, k) with x_{m,k} = 1, k in V_{l,r} (Eq. 8), and
//     Qhat + Q_l(r,k) <= Qbar; a substitute must not be one of the token's
//     routed experts nor a substitute already given to it;
//   cost (Eq. 38) = A[a][s][m] + Cq[r][k] as one fp32 add;
//   argmin (Eq. 43) with the tie rule listed at the top of this file;
//   update (Eq. 44): Qhat += Q_l(r,k*); location = server of slot 0.
// kind: 0 local exact, 1 local substitute, 2 remote exact, 3 remote substitute.
int orc_select(const int32_t* idx, int T, int E, int k, int M, const float* Qtab, const float* Cq,
               const uint64_t* subst, const float* A, const uint32_t* pmask, float qbar,
               const uint8_t* home, uint8_t* loc, float* qhat, int32_t* chosen, uint8_t* server,
               uint8_t* kind) {
  if (E <= 0 || E > 64 || M <= 0 || M > 32 || k <= 0 || k > E) return ORC_BAD_ARG;
  for (int t = 0; t < T; ++t) {
    const int a = home[t];
    const int s = loc[t];
    if (a >= M || s >= M) return ORC_BAD_ARG;
    float q = qhat[t];
    uint64_t taken = 0;
    for (int j = 0; j < k; ++j) taken |= (uint64_t)1 << idx[(int64_t)t * k + j];
    int first_server = -1;
    for (int j = 0; j < k; ++j) {
      const int r = idx[(int64_t)t * k + j];
      if (r < 0 || r >= E) return ORC_BAD_ARG;
      bool have = false;
      float best_cost = 0.0f;
      int best_sub = 0, best_away = 0, best_m = 0, best_k = 0;
      for (int kk = 0; kk < E; ++kk) {
        const bool exact = (kk == r);
        if (!exact) {
          if (!((subst[r] >> kk) & 1u)) continue;           // e_k in R_{l,r}
          if ((taken >> kk) & 1u) continue;                   // distinct experts
          if (!(q + Qtab[r * E + kk] <= qbar)) continue;      // budget, Eq. 40
        }
        for (int m = 0; m < M; ++m) {
          if (!((pmask[kk] >> m) & 1u)) continue;             // x_{m,k} = 1
          const float cost = A[((int64_t)a * M + s) * M + m] + (exact ? 0.0f : Cq[r * E + kk]);
          const int sub = exact ? 0 : 1;
          const int away = (m != s) ? 1 : 0;
          bool better;
          if (!have) better = true;
          else if (cost != best_cost) better = cost < best_cost;
          else if (sub != best_sub) better = sub < best_sub;
          else if (away != best_away) better = away < best_away;
          else if (m != best_m) better = m < best_m;
          else better = kk < best_k;
          if (better) {
            have = true;
            best_cost = cost; best_sub = sub; best_away = away; best_m = m; best_k = kk;
          }
        }
      }
      if (!have) return ORC_BAD_ARG;  // Property 1 violated: target placed nowhere
      chosen[(int64_t)t * k + j] = best_k;
      server[(int64_t)t * k + j] = static_cast<uint8_t>(best_m);
      kind[(int64_t)t * k + j] = static_cast<uint8_t>(2 * best_away + best_sub);
      if (best_sub) {
        taken |= (uint64_t)1 << best_k;
        q = q + Qtab[r * E + best_k];
      }
      if (j == 0) first_server = best_m;
    }
    loc[t] = static_cast<uint8_t>(first_server);
    qhat[t] = q;
  }
  return ORC_OK;
}

// ---------------------------------------------------------------------------
// Token permutation: a stable counting sort of the T*k (token, slot) entries
// by executed expert. offsets[e] = number of entries with expert < e;
// entries of one expert keep their flat (t*k + j) order. row_token[row] = t,
// row_of[t*k + j] = row.
int orc_dispatch(const int32_t* chosen, int T, int k, int E, int32_t* offsets, int32_t* row_token,
                 int32_t* row_of) {
  const int64_t n = (int64_t)T * k;
  std::vector<int64_t> count(E, 0);
  for (int64_t i = 0; i < n; ++i) {
    if (chosen[i] < 0 || chosen[i] >= E) return ORC_BAD_ARG;
    count[chosen[i]]++;
  }
  offsets[0] = 0;
  for (int e = 0; e < E; ++e) offsets[e + 1] = offsets[e] + static_cast<int32_t>(count[e]);
  std::vector<int64_t> next(E);
  for (int e = 0; e < E; ++e) next[e] = offsets[e];
  for (int64_t i = 0; i < n; ++i) {
    int64_t row = next[chosen[i]]++;
    row_token[row] = static_cast<int32_t>(i / k);
    row_of[i] = static_cast<int32_t>(row);
  }
  return ORC_OK;
}

// X_perm[row] = X[row_token[row]] (a copy of bf16 rows).
int orc_gather_rows(const uint16_t* X, const int32_t* row_token, int64_t R, int d, uint16_t* Xp) {
  for (int64_t r = 0; r < R; ++r)
    std::memcpy(Xp + r * d, X + (int64_t)row_token[r] * d, sizeof(uint16_t) * d);
  return ORC_OK;
}

// ---------------------------------------------------------------------------
// SwiGLU expert FFN (the Mixtral-shaped experts of Section VI-A), one row at
// a time, rows given with their expert:
//   g = x W1_e^T, u = x W3_e^T (fp64), h = bf16(fp32(silu(g) * u)),
//   silu(g) = g / (1 + exp(-g)); y = bf16(fp32(h W2_e^T)) (fp64 accumulate).
// W1, W3: [E][dff][d]; W2: [E][d][dff]; all bf16 bits.
int orc_ffn_rows(const uint16_t* Xrows, const int32_t* row_expert, int64_t R, const uint16_t* W1,
                 const uint16_t* W3, const uint16_t* W2, int E, int d, int dff, uint16_t* H,
                 uint16_t* Y) {
  if (E <= 0 || d <= 0 || dff <= 0) return ORC_BAD_ARG;
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t r = 0; r < R; ++r) {
    const int e = row_expert[r];
    if (e < 0 || e >= E) continue;
    const uint16_t* x = Xrows + r * d;
    uint16_t* h = H + r * dff;
    for (int n = 0; n < dff; ++n) {
      const uint16_t* w1 = W1 + ((int64_t)e * dff + n) * d;
      const uint16_t* w3 = W3 + ((int64_t)e * dff + n) * d;
      double g = 0.0, u = 0.0;
      for (int c = 0; c < d; ++c) {
        double xc = bf(x, c);
        g += xc * bf(w1, c);
        u += xc * bf(w3, c);
      }
      double silu = g / (1.0 + std::exp(-g));
      h[n] = float_to_bf16_bits(static_cast<float>(silu * u));
    }
    for (int o = 0; o < d; ++o) {
      const uint16_t* w2 = W2 + ((int64_t)e * d + o) * dff;
      double acc = 0.0;
      for (int n = 0; n < dff; ++n) acc += bf(h, n) * bf(w2, n);
      Y[r * d + o] = float_to_bf16_bits(static_cast<float>(acc));
    }
  }
  return ORC_OK;
}

// Weighted combine: y[t] = bf16(sum_j w[t][j] * Y_perm[row_of[t][j]]), fp64
// accumulation over slots j = 0..k-1.
int orc_combine(const uint16_t* Yp, const int32_t* row_of, const float* w, int T, int k, int d,
                uint16_t* y) {
  for (int t = 0; t < T; ++t)
    for (int c = 0; c < d; ++c) {
      double acc = 0.0;
      for (int j = 0; j < k; ++j) {
        int64_t row = row_of[(int64_t)t * k + j];
        acc += static_cast<double>(w[(int64_t)t * k + j]) * bf(Yp, row * d + c);
      }
      y[(int64_t)t * d + c] = float_to_bf16_bits(static_cast<float>(acc));
    }
  return ORC_OK;
}

// ---------------------------------------------------------------------------
// Residual map between stacked MoE layers. The paper serves Mixtral-8x7B
// (Section VI-A), a stack of pre-norm decoder blocks; without the attention
// half, block l maps the residual stream h_l to h_{l+1} = h_l + y_l, where
// y_l is the MoE layer's output for the input x_l = RMSNorm(h_l) (unit gain):
//   RMSNorm(v)[c] = bf16( v[c] / sqrt( (1/d) sum_c v[c]^2 + eps ) )    (fp64)
//   h_out[t][c]   = bf16( h[t][c] + sum_j w[t][j] Y[row_of[t][j]][c] )  (fp64, slot order)
int orc_rmsnorm(const uint16_t* h, int T, int d, double eps, uint16_t* x) {
  if (T < 0 || d <= 0 || !(eps > 0.0)) return ORC_BAD_ARG;
  for (int t = 0; t < T; ++t) {
    const uint16_t* row = h + (int64_t)t * d;
    double ss = 0.0;
    for (int c = 0; c < d; ++c) ss += bf(row, c) * bf(row, c);
    const double rms = std::sqrt(ss / d + eps);
    for (int c = 0; c < d; ++c)
      x[(int64_t)t * d + c] = float_to_bf16_bits(static_cast<float>(bf(row, c) / rms));
  }
  return ORC_OK;
}

int orc_combine_residual(const uint16_t* Yp, const int32_t* row_of, const float* w,
                         const uint16_t* h, int T, int k, int d, uint16_t* h_out) {
  if (T < 0 || k <= 0 || d <= 0) return ORC_BAD_ARG;
  for (int t = 0; t < T; ++t)
    for (int c = 0; c < d; ++c) {
      double acc = bf(h, (int64_t)t * d + c);
      for (int j = 0; j < k; ++j) {
        const int64_t row = row_of[(int64_t)t * k + j];
        acc += static_cast<double>(w[(int64_t)t * k + j]) * bf(Yp, row * d + c);
      }
      h_out[(int64_t)t * d + c] = float_to_bf16_bits(static_cast<float>(acc));
    }
  return ORC_OK;
}

// ---------------------------------------------------------------------------
// Expert similarity, Eqs. 3-4: H = W_r X_cal^T (fp64), Sim(i,j) = cosine of
// rows i and j of H, fp64 then rounded to fp32; the diagonal is exactly 1 and
// a pair with a zero-norm row has Sim 0. Also returns the fp32 H when Hout is
// not null ([E][N]).
int orc_similarity(const uint16_t* W, const uint16_t* Xc, int E, int d, int64_t N, float* sim,
                   float* Hout) {
  std::vector<double> H((size_t)E * N);
#pragma omp parallel for schedule(static)
  for (int64_t n = 0; n < N; ++n)
    for (int e = 0; e < E; ++e) {
      double acc = 0.0;
      for (int c = 0; c < d; ++c) acc += bf(W, (int64_t)e * d + c) * bf(Xc, n * d + c);
      H[(size_t)e * N + n] = acc;
    }
  if (Hout)
    for (size_t i = 0; i < H.size(); ++i) Hout[i] = static_cast<float>(H[i]);
  std::vector<double> norm(E);
  for (int e = 0; e < E; ++e) {
    double s = 0.0;
    for (int64_t n = 0; n < N; ++n) s += H[(size_t)e * N + n] * H[(size_t)e * N + n];
    norm[e] = std::sqrt(s);
  }
  for (int i = 0; i < E; ++i)
    for (int j = 0; j < E; ++j) {
      if (i == j) { sim[i * E + j] = 1.0f; continue; }
      if (norm[i] == 0.0 || norm[j] == 0.0) { sim[i * E + j] = 0.0f; continue; }
      double dot = 0.0;
      for (int64_t n = 0; n < N; ++n) dot += H[(size_t)i * N + n] * H[(size_t)j * N + n];
      sim[i * E + j] = static_cast<float>(dot / (norm[i] * norm[j]));
    }
  return ORC_OK;
}

// Activation counts n_j of Eq. 5 from given fp32 logits [N][E]: the number
// of tokens whose top-kf experts (rank order of orc_topk) include j.
int orc_expert_counts(const float* logits, int64_t N, int E, int kf, int32_t* count) {
  if (kf <= 0 || kf > E) return ORC_BAD_ARG;
  for (int e = 0; e < E; ++e) count[e] = 0;
  std::vector<int> order(E);
  for (int64_t n = 0; n < N; ++n) {
    const float* l = logits + n * E;
    for (int e = 0; e < E; ++e) order[e] = e;
    std::sort(order.begin(), order.end(),
              [&](int a, int b) { return ranks_before(l[a], a, l[b], b); });
    for (int j = 0; j < kf; ++j) count[order[j]]++;
  }
  return ORC_OK;
}

// Depth-aware threshold, Eq. 6, layers l = 1..N. The formula divides by
// N - 1, so a single-layer model takes theta_single instead.
float orc_theta(int l, int N, double theta_min, double theta_max, double theta_single) {
  if (N <= 1) return static_cast<float>(theta_single);
  double frac = static_cast<double>(N - l) / static_cast<double>(N - 1);
  return static_cast<float>(theta_min + (theta_max - theta_min) * frac);
}

// Greedy representative-cover grouping, Eqs. 24-26 (Alg. 1, grouping loop).
// Experts are visited by decreasing count (ties: lower index). dominant[g] is
// the dominant (centre) of group g.
int orc_group(const float* sim, const int32_t* count, int E, float theta, int32_t* group,
              int32_t* n_groups, int32_t* dominant) {
  std::vector<int> order(E);
  for (int e = 0; e < E; ++e) order[e] = e;
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return count[a] > count[b]; });
  int K = 0;
  for (int pos = 0; pos < E; ++pos) {
    const int j = order[pos];
    int best_g = -1;
    float best_s = 0.0f;
    for (int g = 0; g < K; ++g) {
      float s = sim[j * E + dominant[g]];
      if (best_g < 0 || s > best_s) { best_g = g; best_s = s; }
    }
    if (best_g < 0 || best_s < theta) {
      dominant[K] = j;
      group[j] = K;
      ++K;
    } else {
      group[j] = best_g;
    }
  }
  *n_groups = K;
  return ORC_OK;
}

// Importance, Eqs. 27-28: rho_j = mean of Sim(j,k) over k in j's group (j
// itself included), I_j = alpha_f f_j + alpha_r rho_j, f_j = n_j / sum n.
int orc_importance(const float* sim, const int32_t* count, const int32_t* group, int E,
                   double alpha_f, double alpha_r, double* importance) {
  double total = 0.0;
  for (int e = 0; e < E; ++e) total += count[e];
  for (int j = 0; j < E; ++j) {
    double s = 0.0;
    int size = 0;
    for (int k = 0; k < E; ++k)
      if (group[k] == group[j]) { s += sim[j * E + k]; ++size; }
    double rho = s / size;
    double f = total > 0.0 ? count[j] / total : 0.0;
    importance[j] = alpha_f * f + alpha_r * rho;
  }
  return ORC_OK;
}

// Mandatory placement over L layers, Eqs. 29-31 and Alg. 1's placement loop:
// per layer, experts in order (p desc, I desc, index asc); feasible servers
// b_m + p <= C_m; score = lambda1 b_m / C_m + lambda2 eta (eta = experts of
// the same group already on m in this layer); argmin, ties lower m. Experts
// with no feasible server wait and then go to the server with the largest
// C_m - b_m (ties lower m). b_m accumulates over layers.
// placement: [L][M][E] u8. Returns ORC_CAPACITY if sum C < sum p, or if a
// waiting-list expert overflowed its server.
int orc_place(const int32_t* group, const double* importance, const double* p, int L, int E,
              int M, const double* C, double lambda1, double lambda2, uint8_t* placement,
              double* used) {
  double needed = 0.0, have = 0.0;
  for (int i = 0; i < L * E; ++i) needed += p[i];
  for (int m = 0; m < M; ++m) have += C[m];
  std::memset(placement, 0, (size_t)L * M * E);
  std::vector<double> b(M, 0.0);
  bool overflow = needed > have;
  for (int l = 0; l < L; ++l) {
    const int32_t* g = group + (int64_t)l * E;
    const double* I = importance + (int64_t)l * E;
    const double* pl = p + (int64_t)l * E;
    uint8_t* x = placement + (int64_t)l * M * E;
    std::vector<int> order(E);
    for (int e = 0; e < E; ++e) order[e] = e;
    // p desc, I desc, index asc; a NaN (the importance of NaN similarities)
    // comes after every number, so the comparison is a strict weak order
    auto same = [](double x, double y) { return x == y || (std::isnan(x) && std::isnan(y)); };
    auto above = [](double x, double y) {
      return std::isnan(y) ? !std::isnan(x) : (!std::isnan(x) && x > y);
    };
    std::sort(order.begin(), order.end(), [&](int a, int c) {
      if (!same(pl[a], pl[c])) return above(pl[a], pl[c]);
      if (!same(I[a], I[c])) return above(I[a], I[c]);
      return a < c;
    });
    std::vector<int> waiting;
    for (int j : order) {
      int best = -1;
      double best_score = 0.0;
      for (int m = 0; m < M; ++m) {
        if (!(b[m] + pl[j] <= C[m])) continue;
        int eta = 0;
        for (int k = 0; k < E; ++k)
          if (g[k] == g[j] && x[m * E + k]) ++eta;
        double score = lambda1 * (b[m] / C[m]) + lambda2 * static_cast<double>(eta);
        if (best < 0 || score < best_score) { best = m; best_score = score; }
      }
      if (best < 0) { waiting.push_back(j); continue; }
      x[best * E + j] = 1;
      b[best] += pl[j];
    }
    for (int j : waiting) {
      int best = 0;
      for (int m = 1; m < M; ++m)
        if (C[m] - b[m] > C[best] - b[best]) best = m;
      x[best * E + j] = 1;
      b[best] += pl[j];
      if (b[best] > C[best]) overflow = true;
    }
  }
  for (int m = 0; m < M; ++m) used[m] = b[m];
  return overflow ? ORC_CAPACITY : ORC_OK;
}

// ---------------------------------------------------------------------------
// Importance-aware redundant deployment, Section IV-C (Eqs. 32-35, Alg. 1),
// over all layers after the mandatory placement. y[m][l][g]
// (Eq. 32) is 1 when server m hosts an expert of group g in layer l. A
// candidate replica of expert j of layer l on server m has the benefit
// B = pi_m * I_l^j * (1 - y[m][l][g(j)]) / p_l^j (Eq. 33), and fits when
// b_m + p_l^j <= C_m (Eq. 35). Greedy: each round recomputes every benefit,
// deploys the largest one that fits (ties: lower layer, then lower server,
// then lower expert), updates y and b_m, and stops when no fitting candidate
// has a positive benefit. placement [L][M][E] and used [M] are updated in
// place; replicas [M] counts the replicas per server. pi [M]: the share of
// the tokens whose trajectory reaches each server.
int orc_replicate(const int32_t* group, const double* importance, const double* p, int L, int E,
                  int M, const double* C, const double* pi, uint8_t* placement, double* used,
                  int32_t* replicas) {
  for (int i = 0; i < L * E; ++i)
    if (!(p[i] > 0.0) || group[i] < 0 || group[i] >= E) return ORC_BAD_ARG;
  // Eq. 32 from the mandatory placement
  std::vector<uint8_t> y((size_t)M * L * E, 0);
  for (int l = 0; l < L; ++l)
    for (int m = 0; m < M; ++m)
      for (int j = 0; j < E; ++j)
        if (placement[((size_t)l * M + m) * E + j])
          y[((size_t)m * L + l) * E + group[l * E + j]] = 1;
  for (int m = 0; m < M; ++m) replicas[m] = 0;
  for (;;) {
    int bl = -1, bm = -1, bj = -1;
    double bb = 0.0;
    for (int l = 0; l < L; ++l)
      for (int m = 0; m < M; ++m)
        for (int j = 0; j < E; ++j) {
          const int g = group[l * E + j];
          const double cover = 1.0 - static_cast<double>(y[((size_t)m * L + l) * E + g]);
          const double benefit = pi[m] * importance[l * E + j] * cover / p[l * E + j];
          if (!(benefit > 0.0)) continue;
          if (!(used[m] + p[l * E + j] <= C[m])) continue;
          if (bl < 0 || benefit > bb) { bl = l; bm = m; bj = j; bb = benefit; }
        }
    if (bl < 0) break;
    placement[((size_t)bl * M + bm) * E + bj] = 1;
    used[bm] += p[bl * E + bj];
    y[((size_t)bm * L + bl) * E + group[bl * E + bj]] = 1;
    replicas[bm]++;
  }
  return ORC_OK;
}

// ---------------------------------------------------------------------------
// Edge cost of the selection records of L layers (Section III-D/E): a token
// starts at its home server a (Eq. 36); at layer l each slot j executed on
// server m_j pays the transfer of Eqs. 13-14 from the token's location s_l
// when m_j != s_l, z / B[s_l][m_j] + tau[s_l][m_j], plus the compute of
// Eq. 15, c / F[m_j]; the location after the layer is the server of slot 0
// (Eq. 44). delay[t] = sum over layers and slots (Eqs. 16-17, one token per
// user), loss[t] = the substitution loss Q_l(r, k) of every substituted slot
// (Eqs. 18-20; Qtab [L][E][E], the fp32 values the selection uses), moves[t]
// = the number of transfers. fp64, one running sum per token in (l, j) order.
int orc_trajectory_cost(const int32_t* target, const int32_t* chosen, const uint8_t* server,
                        const uint8_t* home, int L, int T, int k, int E, int M, const double* F,
                        const double* B, const double* tau, double z, double c, const float* Qtab,
                        double* delay, double* loss, int32_t* moves) {
  for (int t = 0; t < T; ++t) {
    int s = home[t];
    if (s >= M) return ORC_BAD_ARG;
    double d = 0.0, q = 0.0;
    int n = 0;
    for (int l = 0; l < L; ++l) {
      int next = s;
      for (int j = 0; j < k; ++j) {
        const size_t i = ((size_t)l * T + t) * k + j;
        const int r = target[i], kk = chosen[i], m = server[i];
        if (r < 0 || r >= E || kk < 0 || kk >= E || m >= M) return ORC_BAD_ARG;
        double trans = 0.0;
        if (m != s) {
          trans = z / B[s * M + m] + tau[s * M + m];
          ++n;
        }
        const double comp = c / F[m];
        d = d + (trans + comp);
        if (kk != r) q = q + static_cast<double>(Qtab[((size_t)l * E + r) * E + kk]);
        if (j == 0) next = m;
      }
      s = next;
    }
    delay[t] = d;
    loss[t] = q;
    moves[t] = n;
  }
  return ORC_OK;
}

// Normalised utility (Eq. 23) and weight adaptation (Eq. 45) over T users
// (one token each): T~ = delay / delay_ref (delay_ref: the same tokens under
// pure exact execution on the same deployment), Q~ = loss / qmax;
// U = omega_T sum T~ + omega_Q sum Q~; Tbar, Qbar the means;
// omega_Q' = clamp(omega_Q + kappa (Qbar - Tbar), 0, 1), omega_T' = 1 - omega_Q'.
// out[5] = {U, Tbar, Qbar, omega_T', omega_Q'}.
int orc_utility(const double* delay, const double* delay_ref, const double* loss, int T,
                double qmax, double omega_T, double omega_Q, double kappa, double* out) {
  if (T <= 0 || !(qmax > 0.0)) return ORC_BAD_ARG;
  double st = 0.0, sq = 0.0;
  for (int t = 0; t < T; ++t) {
    if (!(delay_ref[t] > 0.0)) return ORC_BAD_ARG;
    st += delay[t] / delay_ref[t];
    sq += loss[t] / qmax;
  }
  const double tbar = st / T, qbar = sq / T;
  double wq = omega_Q + kappa * (qbar - tbar);
  wq = std::min(1.0, std::max(0.0, wq));
  out[0] = omega_T * st + omega_Q * sq;
  out[1] = tbar;
  out[2] = qbar;
  out[3] = 1.0 - wq;
  out[4] = wq;
  return ORC_OK;
}

// ---------------------------------------------------------------------------
// Expert transition statistics, Eq. 41, from calibration logits [N][L][E]:
// for each token, every pair (k in top-kf of layer l, k' in top-kf of layer
// l+1) counts one transition k -> k' (the paper has one target per token; with
// top-k each routed pair counts). P_l(k -> k') = n / sum_k'' n(k -> k''), fp64
// then rounded to fp32; a row with no transitions is all zero.
int orc_transitions(const float* logits, int64_t N, int L, int E, int kf, int32_t* count,
                    float* P) {
  if (L < 2 || E <= 0 || kf <= 0 || kf > E) return ORC_BAD_ARG;
  std::memset(count, 0, sizeof(int32_t) * (size_t)(L - 1) * E * E);
  std::vector<int> cur(kf), nxt(kf), order(E);
  auto topk = [&](const float* l, std::vector<int>& out) {
    for (int e = 0; e < E; ++e) order[e] = e;
    std::sort(order.begin(), order.end(),
              [&](int a, int b) { return ranks_before(l[a], a, l[b], b); });
    for (int j = 0; j < kf; ++j) out[j] = order[j];
  };
  for (int64_t n = 0; n < N; ++n) {
    topk(logits + (n * L) * E, cur);
    for (int l = 0; l + 1 < L; ++l) {
      topk(logits + (n * L + l + 1) * E, nxt);
      for (int a : cur)
        for (int b : nxt) count[((size_t)l * E + a) * E + b]++;
      cur = nxt;
    }
  }
  for (int l = 0; l + 1 < L; ++l)
    for (int a = 0; a < E; ++a) {
      double row = 0.0;
      for (int b = 0; b < E; ++b) row += count[((size_t)l * E + a) * E + b];
      for (int b = 0; b < E; ++b)
        P[((size_t)l * E + a) * E + b] =
            row > 0.0 ? static_cast<float>(count[((size_t)l * E + a) * E + b] / row) : 0.0f;
    }
  return ORC_OK;
}

// One layer's selection tables as the look-ahead reads them (see orc_tables).
struct OrcTab {
  const float* Qtab;
  const float* Cq;
  const uint64_t* subst;
  const float* A;
  const uint32_t* pmask;
};

// Look-ahead cost-to-go of Eq. 42 with h future layers (h >= 1): being at
// server m after executing expert kx at layer l with accumulated loss qacc,
//   Phi^(h) = sum_{k'} P_l(kx -> k') * min over the feasible pairs (m', k'')
//             of target k' at layer l+1 (Eq. 40, from server m) of
//             [ g_{l+1}(m', k'' | s = m) + Phi^(h-1)_{l+1}(m', k'') ],
// with Phi^(0) = 0. In the future layers a token has the single target k'
// (no distinct-expert rule) and the same home server a; the loss of a
// future substitute adds to qacc. fp32 arithmetic: each product and sum is
// one rounded fp32 operation, k' in ascending order.
float orc_phi(int h, const OrcTab* tabs, const float* P, int E, int M, int a, int m, int kx,
              float qacc, float qbar) {
  if (h <= 0) return 0.0f;
  const OrcTab& t1 = tabs[1];
  float acc = 0.0f;
  for (int kt = 0; kt < E; ++kt) {
    const float p = P[(size_t)kx * E + kt];
    if (p == 0.0f) continue;
    float best = INFINITY;
    for (int kk = 0; kk < E; ++kk) {
      const bool exact = (kk == kt);
      float q2 = qacc;
      if (!exact) {
        if (!((t1.subst[kt] >> kk) & 1u)) continue;
        if (!(qacc + t1.Qtab[kt * E + kk] <= qbar)) continue;
        q2 = qacc + t1.Qtab[kt * E + kk];
      }
      for (int m2 = 0; m2 < M; ++m2) {
        if (!((t1.pmask[kk] >> m2) & 1u)) continue;
        float c = t1.A[((int64_t)a * M + m) * M + m2] + (exact ? 0.0f : t1.Cq[kt * E + kk]);
        if (h > 1) c = c + orc_phi(h - 1, tabs + 1, P + (size_t)E * E, E, M, a, m2, kk, q2, qbar);
        if (c < best) best = c;
      }
    }
    const float term = p * best;
    acc = acc + term;
  }
  return acc;
}

// Alg. 2 with horizon H (Eq. 43): as orc_select, but each candidate (m, k)
// of layer l costs g_l(m, k) + Phi^(H-1)(m, k) (one fp32 add), the cost-to-go
// computed with the tables of layers l+1 .. l+H-1 (tabs[1..H-1]) and the
// transition matrices P_l .. P_{l+H-2} (P, [H-1][E][E]). H = 1 is orc_select.
int orc_select_lookahead(const int32_t* idx, int T, int E, int k, int M, int H, const float* Qtab,
                         const float* Cq, const uint64_t* subst, const float* A,
                         const uint32_t* pmask, const float* const* nQtab, const float* const* nCq,
                         const uint64_t* const* nsubst, const float* const* nA,
                         const uint32_t* const* npmask, const float* P, float qbar,
                         const uint8_t* home, uint8_t* loc, float* qhat, int32_t* chosen,
                         uint8_t* server, uint8_t* kind) {
  if (E <= 0 || E > 64 || M <= 0 || M > 32 || k <= 0 || k > E || H < 1 || H > 4) return ORC_BAD_ARG;
  std::vector<OrcTab> tabs(H);
  tabs[0] = OrcTab{Qtab, Cq, subst, A, pmask};
  for (int h = 1; h < H; ++h) tabs[h] = OrcTab{nQtab[h - 1], nCq[h - 1], nsubst[h - 1], nA[h - 1], npmask[h - 1]};
  for (int t = 0; t < T; ++t) {
    const int a = home[t];
    const int s = loc[t];
    if (a >= M || s >= M) return ORC_BAD_ARG;
    float q = qhat[t];
    uint64_t taken = 0;
    for (int j = 0; j < k; ++j) taken |= (uint64_t)1 << idx[(int64_t)t * k + j];
    int first_server = -1;
    for (int j = 0; j < k; ++j) {
      const int r = idx[(int64_t)t * k + j];
      if (r < 0 || r >= E) return ORC_BAD_ARG;
      bool have = false;
      float best_cost = 0.0f;
      int best_sub = 0, best_away = 0, best_m = 0, best_k = 0;
      for (int kk = 0; kk < E; ++kk) {
        const bool exact = (kk == r);
        if (!exact) {
          if (!((subst[r] >> kk) & 1u)) continue;
          if ((taken >> kk) & 1u) continue;
          if (!(q + Qtab[r * E + kk] <= qbar)) continue;
        }
        const float qn = exact ? q : q + Qtab[r * E + kk];
        for (int m = 0; m < M; ++m) {
          if (!((pmask[kk] >> m) & 1u)) continue;
          float cost = A[((int64_t)a * M + s) * M + m] + (exact ? 0.0f : Cq[r * E + kk]);
          cost = cost + orc_phi(H - 1, tabs.data(), P, E, M, a, m, kk, qn, qbar);
          const int sub = exact ? 0 : 1;
          const int away = (m != s) ? 1 : 0;
          bool better;
          if (!have) better = true;
          else if (cost != best_cost) better = cost < best_cost;
          else if (sub != best_sub) better = sub < best_sub;
          else if (away != best_away) better = away < best_away;
          else if (m != best_m) better = m < best_m;
          else better = kk < best_k;
          if (better) {
            have = true;
            best_cost = cost; best_sub = sub; best_away = away; best_m = m; best_k = kk;
          }
        }
      }
      if (!have) return ORC_BAD_ARG;
      chosen[(int64_t)t * k + j] = best_k;
      server[(int64_t)t * k + j] = static_cast<uint8_t>(best_m);
      kind[(int64_t)t * k + j] = static_cast<uint8_t>(2 * best_away + best_sub);
      if (best_sub) {
        taken |= (uint64_t)1 << best_k;
        q = q + Qtab[r * E + best_k];
      }
      if (j == 0) first_server = best_m;
    }
    loc[t] = static_cast<uint8_t>(first_server);
    qhat[t] = q;
  }
  return ORC_OK;
}

// Local group coverage, Eq. 32 (indices read as y_{m,l,g} = 1 when server m
// hosts at least one expert of group g in layer l). cover: [M][K].
int orc_coverage(const uint8_t* placement_l, const int32_t* group_l, int E, int M, int K,
                 uint8_t* cover) {
  std::memset(cover, 0, (size_t)M * K);
  for (int m = 0; m < M; ++m)
    for (int e = 0; e < E; ++e)
      if (placement_l[m * E + e]) cover[m * K + group_l[e]] = 1;
  return ORC_OK;
}

// Threads of the oracle's OpenMP loops (only over independent tokens and
// rows, so the results do not depend on it): the count the next parallel
// region uses, and a setter (n >= 1) for timing the oracle on fewer cores.
int orc_threads(void) { return omp_get_max_threads(); }
int orc_set_threads(int n) {
  if (n < 1) return ORC_BAD_ARG;
  omp_set_num_threads(n);
  return ORC_OK;
}

}  // extern "C"
