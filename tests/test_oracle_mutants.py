"""The pins must catch plausible mistakes in the oracle.

Each case plants one mistake (a dropped term, a wrong sign or index, a
transposed operand, a wrong tie rule) in a temporary copy of the oracle's
source, builds it, loads it in place of the real oracle, and runs the pin
tests against it: at least one pin must fail. The real oracle is never
modified.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "ordermoe_oracle.cpp")

# anchors inside orc_select_lookahead (each occurs once in the source)
LA_TIE = ("cost = cost + orc_phi(H - 1, tabs.data(), P, E, M, a, m, kk, qn, qbar);\n"
          "          const int sub = exact ? 0 : 1;\n          const int away = (m != s) ? 1 : 0;\n"
          "          bool better;\n          if (!have) better = true;\n"
          "          else if (cost != best_cost) better = cost < best_cost;\n"
          "          else if (sub != best_sub) better = sub < best_sub;")
LA_END = ("      if (!have) return ORC_BAD_ARG;\n      chosen[(int64_t)t * k + j] = best_k;\n"
          "      server[(int64_t)t * k + j] = static_cast<uint8_t>(best_m);\n"
          "      kind[(int64_t)t * k + j] = static_cast<uint8_t>(2 * best_away + best_sub);\n"
          "      if (best_sub) {\n        taken |= (uint64_t)1 << best_k;\n"
          "        q = q + Qtab[r * E + best_k];\n      }\n      if (j == 0) first_server = best_m;")
LA_DIST = ("          if ((taken >> kk) & 1u) continue;\n"
           "          if (!(q + Qtab[r * E + kk] <= qbar)) continue;\n        }\n        const float qn")

# (name, original text, planted mistake)
MUTANTS = [
    ("router: W transposed", "acc += bf(X, (int64_t)t * d + c) * bf(W, (int64_t)e * d + c);",
     "acc += bf(X, (int64_t)t * d + c) * bf(W, (int64_t)c * E + e);"),
    ("topk: ties to higher index", "return ia < ib;", "return ia > ib;"),
    ("topk: no renormalisation", "renorm ? p[order[j]] / ssel : p[order[j]]", "p[order[j]]"),
    ("Eq. 18: sign of Sim", "q = 0.5f * (1.0f - std::min(s, 1.0f));", "q = 0.5f * (1.0f + std::min(s, 1.0f));"),
    ("Eq. 38: quality term not divided by Qbar",
     "omega_Q * static_cast<double>(q) / static_cast<double>(qbar)", "omega_Q * static_cast<double>(q)"),
    ("Eq. 7: threshold ignored", "group[k] == group[r] && s >= theta", "group[k] == group[r]"),
    ("Eq. 7: group ignored", "group[k] == group[r] && s >= theta", "s >= theta"),
    ("Eq. 37: latency dropped", "z / B[s * M + m] + tau[s * M + m]", "z / B[s * M + m]"),
    ("Eq. 37: compute on the source server", "double comp = c / F[m];", "double comp = c / F[s];"),
    ("Eq. 38: d_ref of the executing server", "double dref = c / F[a];", "double dref = c / F[0];"),
    ("Eq. 40: budget ignored", "if (!(q + Qtab[r * E + kk] <= qbar)) continue;", ""),
    ("distinct experts ignored", "if ((taken >> kk) & 1u) continue;", ""),
    ("tie: remote preferred", "better = away < best_away;", "better = away > best_away;"),
    ("Eq. 44: loss not accumulated", "q = q + Qtab[r * E + best_k];", ""),
    ("Eq. 44: location from the last slot", "if (j == 0) first_server = best_m;", "first_server = best_m;"),
    ("permutation not stable", "row_token[row] = static_cast<int32_t>(i / k);",
     "row_token[row] = static_cast<int32_t>((n - 1 - i) / k);"),
    ("FFN: gate and up swapped", "double silu = g / (1.0 + std::exp(-g));\n      h[n] = float_to_bf16_bits(static_cast<float>(silu * u));",
     "double silu = u / (1.0 + std::exp(-u));\n      h[n] = float_to_bf16_bits(static_cast<float>(silu * g));"),
    ("FFN: W2 transposed", "W2 + ((int64_t)e * d + o) * dff", "W2 + (int64_t)e * d * dff + o"),
    ("combine: weights dropped", "acc += static_cast<double>(w[(int64_t)t * k + j]) * bf(Yp, row * d + c);",
     "acc += bf(Yp, row * d + c);"),
    ("RMSNorm: sum of squares not divided by d", "std::sqrt(ss / d + eps)", "std::sqrt(ss + eps)"),
    ("RMSNorm: square root dropped", "std::sqrt(ss / d + eps)", "(ss / d + eps)"),
    ("residual combine: residual dropped", "double acc = bf(h, (int64_t)t * d + c);", "double acc = 0.0;"),
    ("residual combine: weights dropped",
     "acc += static_cast<double>(w[(int64_t)t * k + j]) * bf(Yp, row * d + c);\n      }\n      h_out",
     "acc += bf(Yp, row * d + c);\n      }\n      h_out"),
    ("Eq. 4: not normalised", "dot / (norm[i] * norm[j])", "dot"),
    ("Eq. 24: threshold inclusive", "best_s < theta", "best_s <= theta"),
    ("Eq. 25: argmax ties to the later dominant", "if (best_g < 0 || s > best_s)", "if (best_g < 0 || s >= best_s)"),
    ("Eq. 25: -0 ranked below +0", "if (best_g < 0 || s > best_s)",
     "if (best_g < 0 || s > best_s || (s == 0.0f && best_s == 0.0f && std::signbit(best_s) && !std::signbit(s)))"),
    ("Eq. 27: representativeness over all experts", "if (group[k] == group[j]) { s += sim[j * E + k]; ++size; }",
     "{ s += sim[j * E + k]; ++size; }"),
    ("Eq. 30: dispersion term dropped", "lambda2 * static_cast<double>(eta)", "0.0"),
    ("Eq. 29: capacity ignored", "if (!(b[m] + pl[j] <= C[m])) continue;", ""),
    ("Eq. 32: coverage not updated after a replica",
     "y[((size_t)bm * L + bl) * E + group[bl * E + bj]] = 1;", ""),
    ("Eq. 33: coverage term dropped",
     "const double cover = 1.0 - static_cast<double>(y[((size_t)m * L + l) * E + g]);",
     "const double cover = 1.0;"),
    ("Eq. 33: benefit not per unit memory", "* cover / p[l * E + j];", "* cover;"),
    ("Eq. 33: pi dropped", "const double benefit = pi[m] * importance", "const double benefit = 1.0 * importance"),
    ("Eq. 35: capacity ignored", "if (!(used[m] + p[l * E + j] <= C[m])) continue;", ""),
    ("Eq. 35: used memory not updated", "used[bm] += p[bl * E + bj];", ""),
    ("redundancy: ties to the later candidate", "if (bl < 0 || benefit > bb) { bl = l;",
     "if (bl < 0 || benefit >= bb) { bl = l;"),
    ("Eq. 14: simulator transfer from the home server",
     "trans = z / B[s * M + m] + tau[s * M + m];\n          ++n;",
     "trans = z / B[home[t] * M + m] + tau[home[t] * M + m];\n          ++n;"),
    ("Eq. 13: simulator latency dropped", "trans = z / B[s * M + m] + tau[s * M + m];\n          ++n;",
     "trans = z / B[s * M + m];\n          ++n;"),
    ("Eq. 15: simulator compute on the source server", "const double comp = c / F[m];",
     "const double comp = c / F[s];"),
    ("Eq. 44: simulator location from the last slot", "if (j == 0) next = m;", "next = m;"),
    ("Eq. 19: loss of the substitute's own row", "Qtab[((size_t)l * E + r) * E + kk]",
     "Qtab[((size_t)l * E + kk) * E + r]"),
    ("Eq. 23: weights swapped", "out[0] = omega_T * st + omega_Q * sq;", "out[0] = omega_Q * st + omega_T * sq;"),
    ("Eq. 45: direction flipped", "omega_Q + kappa * (qbar - tbar)", "omega_Q + kappa * (tbar - qbar)"),
    ("Eq. 45: no projection", "wq = std::min(1.0, std::max(0.0, wq));", ""),
    ("Eq. 6: threshold runs the wrong way over the layers",
     "double frac = static_cast<double>(N - l) / static_cast<double>(N - 1);",
     "double frac = static_cast<double>(l - 1) / static_cast<double>(N - 1);"),
    ("placement order: importance ascending", "if (!same(I[a], I[c])) return above(I[a], I[c]);",
     "if (!same(I[a], I[c])) return above(I[c], I[a]);"),
    ("waiting list to the fullest server", "if (C[m] - b[m] > C[best] - b[best]) best = m;",
     "if (C[m] - b[m] < C[best] - b[best]) best = m;"),
    ("Eq. 34: ties to the later layer", "if (bl < 0 || benefit > bb) { bl = l; bm = m; bj = j; bb = benefit; }",
     "if (bl < 0 || benefit >= bb) { if (benefit == bb && l == bl) continue; bl = l; bm = m; bj = j; bb = benefit; }"),
    ("Eq. 45: sums instead of means", "const double tbar = st / T, qbar = sq / T;",
     "const double tbar = st, qbar = sq;"),
    ("Eq. 42: future substitutes ignore the budget",
     "if (!(qacc + t1.Qtab[kt * E + kk] <= qbar)) continue;", ""),
    ("Eq. 37: selection transfer measured from the home server",
     "const float cost = A[((int64_t)a * M + s) * M + m] + (exact ? 0.0f : Cq[r * E + kk]);",
     "const float cost = A[((int64_t)a * M + a) * M + m] + (exact ? 0.0f : Cq[r * E + kk]);"),
    ("Eq. 38: delay weight dropped", "double num = omega_T * dl;", "double num = dl;"),
    ("Eq. 5: counts from the top-1 only", "for (int j = 0; j < kf; ++j) count[order[j]]++;",
     "count[order[0]]++;"),
    ("Eq. 41: normalised over the wrong index",
     "for (int b = 0; b < E; ++b) row += count[((size_t)l * E + a) * E + b];",
     "for (int b = 0; b < E; ++b) row += count[((size_t)l * E + b) * E + a];"),
    ("Eq. 32: coverage of experts instead of groups", "cover[m * K + group_l[e]] = 1;",
     "cover[m * K + (e % K)] = 1;"),
    ("Eq. 28: weights swapped", "importance[j] = alpha_f * f + alpha_r * rho;",
     "importance[j] = alpha_r * f + alpha_f * rho;"),
    ("Eq. 41: transitions of the same layer", "topk(logits + (n * L + l + 1) * E, nxt);",
     "topk(logits + (n * L + l) * E, nxt);"),
    ("Eq. 42: transition from the target, not the executed expert",
     "cost = cost + orc_phi(H - 1, tabs.data(), P, E, M, a, m, kk, qn, qbar);",
     "cost = cost + orc_phi(H - 1, tabs.data(), P, E, M, a, m, r, qn, qbar);"),
    ("Eq. 42: next move measured from the home server",
     "float c = t1.A[((int64_t)a * M + m) * M + m2]", "float c = t1.A[((int64_t)a * M + a) * M + m2]"),
    ("Eq. 42: probabilities dropped", "const float term = p * best;", "const float term = best;"),
    ("Eq. 42: deeper levels reuse the first transition matrix",
     "orc_phi(h - 1, tabs + 1, P + (size_t)E * E, E, M, a, m2, kk, q2, qbar)",
     "orc_phi(h - 1, tabs + 1, P, E, M, a, m2, kk, q2, qbar)"),
    ("Eq. 42: deeper levels reuse the next layer's tables",
     "orc_phi(h - 1, tabs + 1, P + (size_t)E * E, E, M, a, m2, kk, q2, qbar)",
     "orc_phi(h - 1, tabs, P + (size_t)E * E, E, M, a, m2, kk, q2, qbar)"),
    ("Eq. 43: cost-to-go ignored",
     "cost = cost + orc_phi(H - 1, tabs.data(), P, E, M, a, m, kk, qn, qbar);", ""),
    ("Eq. 40: budget strict", "if (!(q + Qtab[r * E + kk] <= qbar)) continue;      // budget",
     "if (!(q + Qtab[r * E + kk] < qbar)) continue;      // budget"),
    ("Eq. 42: budget strict", "if (!(qacc + t1.Qtab[kt * E + kk] <= qbar)) continue;",
     "if (!(qacc + t1.Qtab[kt * E + kk] < qbar)) continue;"),
    ("Eq. 42: the most expensive candidate", "if (c < best) best = c;",
     "if (best == INFINITY || c > best) best = c;"),
    ("execution type bits swapped", "2 * best_away + best_sub", "2 * best_sub + best_away"),
    ("tie: substitute before the exact expert", "else if (sub != best_sub) better = sub < best_sub;",
     "else if (sub != best_sub) better = sub > best_sub;"),
    ("tie: higher server", "else if (m != best_m) better = m < best_m;",
     "else if (m != best_m) better = m > best_m;"),
    ("tie: higher expert", "else better = kk < best_k;", "else better = kk > best_k;"),
    ("distinct experts: a substitute not marked taken", "taken |= (uint64_t)1 << best_k;", ""),
    ("Eq. 29: capacity strict", "if (!(b[m] + pl[j] <= C[m])) continue;",
     "if (!(b[m] + pl[j] < C[m])) continue;"),
    ("Eq. 30: lambda1 dropped", "lambda1 * (b[m] / C[m])", "(b[m] / C[m])"),
    ("Eq. 30: dispersion over every expert", "if (g[k] == g[j] && x[m * E + k]) ++eta;",
     "if (x[m * E + k]) ++eta;"),
    ("Eq. 31: argmin ties to the later server", "if (best < 0 || score < best_score)",
     "if (best < 0 || score <= best_score)"),
    ("waiting list ties to the later server", "if (C[m] - b[m] > C[best] - b[best]) best = m;",
     "if (C[m] - b[m] >= C[best] - b[best]) best = m;"),
    ("Eq. 27: mean over all experts' count", "double rho = s / size;", "double rho = s / E;"),
    ("Eq. 28: frequency not normalised", "count[j] / total : 0.0", "count[j] : 0.0"),
    ("Eq. 7: threshold strict", "if (k != r && group[k] == group[r] && s >= theta) bits",
     "if (k != r && group[k] == group[r] && s > theta) bits"),
    ("Eq. 18: Sim not clamped", "q = 0.5f * (1.0f - std::min(s, 1.0f));", "q = 0.5f * (1.0f - s);"),
    ("Eq. 37: compute dropped on the local server", "double dl = comp;", "double dl = 0.0;"),
    ("Eqs. 15-16: simulator compute dropped", "d = d + (trans + comp);", "d = d + trans;"),
    ("Eq. 23: delay not normalised", "st += delay[t] / delay_ref[t];", "st += delay[t];"),
    ("Eq. 23: loss not normalised", "sq += loss[t] / qmax;", "sq += loss[t];"),
    ("Eq. 45: omega_T not the complement", "out[3] = 1.0 - wq;", "out[3] = omega_T;"),
    ("Eq. 41: top-1 pairs only", "for (int b : nxt) count[((size_t)l * E + a) * E + b]++;",
     "if (a == cur[0]) count[((size_t)l * E + a) * E + nxt[0]]++;"),
    ("Eq. 41: every layer paired with layer 0", "      cur = nxt;\n", "\n"),
    ("Eq. 42: transition matrix transposed", "const float p = P[(size_t)kx * E + kt];",
     "const float p = P[(size_t)kt * E + kx];"),
    ("Eq. 6: one layer takes theta_max", "if (N <= 1) return static_cast<float>(theta_single);",
     "if (N <= 1) return static_cast<float>(theta_max);"),
    ("RMSNorm: eps dropped", "std::sqrt(ss / d + eps)", "std::sqrt(ss / d)"),
    ("SiLU: sign of the exponent", "double silu = g / (1.0 + std::exp(-g));",
     "double silu = g / (1.0 + std::exp(g));"),
    ("Eq. 33: importance dropped", "const double benefit = pi[m] * importance[l * E + j] * cover",
     "const double benefit = pi[m] * 1.0 * cover"),
    ("Eq. 35: capacity strict", "if (!(used[m] + p[l * E + j] <= C[m])) continue;",
     "if (!(used[m] + p[l * E + j] < C[m])) continue;"),
    ("grouping: visited by increasing count", "return count[a] > count[b]; });",
     "return count[a] < count[b]; });"),
    ("grouping: equal counts visited from the higher index",
     "std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return count[a] > count[b]; });",
     "std::sort(order.begin(), order.end(), "
     "[&](int a, int b) { return count[a] > count[b] || (count[a] == count[b] && a > b); });"),
    ("Eq. 4: a zero-norm pair gets Sim 1", "{ sim[i * E + j] = 0.0f; continue; }",
     "{ sim[i * E + j] = 1.0f; continue; }"),
    ("permutation: slot instead of token", "row_token[row] = static_cast<int32_t>(i / k);",
     "row_token[row] = static_cast<int32_t>(i % k);"),
    ("gather: the first token's row everywhere", "X + (int64_t)row_token[r] * d",
     "X + (int64_t)row_token[0] * d"),
    ("Eq. 23: utility from the means", "out[0] = omega_T * st + omega_Q * sq;",
     "out[0] = omega_T * tbar + omega_Q * qbar;"),
    ("Eq. 14: transfers not counted", "trans = z / B[s * M + m] + tau[s * M + m];\n          ++n;",
     "trans = z / B[s * M + m] + tau[s * M + m];"),
    ("Eq. 32: unplaced experts cover their group",
     "if (placement_l[m * E + e]) cover[m * K + group_l[e]] = 1;", "cover[m * K + group_l[e]] = 1;"),
    ("Eq. 42: future budget from the loss before the substitute",
     "const float qn = exact ? q : q + Qtab[r * E + kk];", "const float qn = q;"),
    ("softmax: renormalised over all experts", "for (int j = 0; j < k; ++j) ssel += p[order[j]];",
     "for (int j = 0; j < E; ++j) ssel += p[order[j]];"),
    ("Eq. 37: links read transposed", "double trans = z / B[s * M + m] + tau[s * M + m];",
     "double trans = z / B[m * M + s] + tau[m * M + s];"),
    ("Eq. 41: an empty row spread uniformly",
     "row > 0.0 ? static_cast<float>(count[((size_t)l * E + a) * E + b] / row) : 0.0f;",
     "row > 0.0 ? static_cast<float>(count[((size_t)l * E + a) * E + b] / row) : 1.0f / E;"),
    ("Eq. 4: the diagonal computed, not 1", "if (i == j) { sim[i * E + j] = 1.0f; continue; }", ""),
    ("Eq. 29: load not updated", "      x[best * E + j] = 1;\n      b[best] += pl[j];\n    }",
     "      x[best * E + j] = 1;\n    }"),
    ("waiting list: overflow not reported", "if (b[best] > C[best]) overflow = true;", ""),
    ("Eq. 34: replicas not counted", "replicas[bm]++;", ""),
    ("Eq. 45: projected onto [0, inf) only", "wq = std::min(1.0, std::max(0.0, wq));",
     "wq = std::max(0.0, wq);"),
    ("Eq. 45: projected onto (-inf, 1] only", "wq = std::min(1.0, std::max(0.0, wq));",
     "wq = std::min(1.0, wq);"),
    ("topk: larger logits ranked last", "  if (a != b) return a > b;\n  return ia < ib;",
     "  if (a != b) return a < b;\n  return ia < ib;"),
    ("softmax: not normalised", "for (int e = 0; e < E; ++e) p[e] /= s;", ""),
    ("topk: a NaN logit accepted", "if (std::isnan(l[e])) return ORC_NAN;", ""),
    ("placement order: size ascending", "if (!same(pl[a], pl[c])) return above(pl[a], pl[c]);",
     "if (!same(pl[a], pl[c])) return above(pl[c], pl[a]);"),
    ("placement order: equal keys by the higher index", "      return a < c;\n    });",
     "      return a > c;\n    });"),
    ("Eq. 20: loss read from the exact expert's entry",
     "if (kk != r) q = q + static_cast<double>(Qtab[((size_t)l * E + r) * E + kk]);",
     "if (kk != r) q = q + static_cast<double>(Qtab[((size_t)l * E + r) * E + r]);"),
    ("Eq. 23: means over T - 1", "const double tbar = st / T, qbar = sq / T;",
     "const double tbar = st / (T - 1 > 0 ? T - 1 : 1), qbar = sq / (T - 1 > 0 ? T - 1 : 1);"),
    ("Eq. 28: no activations give frequency 1", "double f = total > 0.0 ? count[j] / total : 0.0;",
     "double f = total > 0.0 ? count[j] / total : 1.0;"),
    ("Eq. 6: theta_min and theta_max swapped",
     "return static_cast<float>(theta_min + (theta_max - theta_min) * frac);",
     "return static_cast<float>(theta_max + (theta_min - theta_max) * frac);"),
    ("router: fp32 running sum",
     "      double acc = 0.0;\n      for (int c = 0; c < d; ++c) acc += bf(X, (int64_t)t * d + c)",
     "      float acc = 0.0f;\n      for (int c = 0; c < d; ++c) acc += bf(X, (int64_t)t * d + c)"),
    ("combine: fp32 running sum",
     "      double acc = 0.0;\n      for (int j = 0; j < k; ++j) {\n        int64_t row",
     "      float acc = 0.0f;\n      for (int j = 0; j < k; ++j) {\n        int64_t row"),
    ("Eq. 3: similarity's H as an fp32 running sum",
     "      double acc = 0.0;\n      for (int c = 0; c < d; ++c) acc += bf(W, (int64_t)e * d + c) * bf(Xc, n * d + c);",
     "      float acc = 0.0f;\n      for (int c = 0; c < d; ++c) acc += bf(W, (int64_t)e * d + c) * bf(Xc, n * d + c);"),
    ("RMSNorm: mean over d - 1", "std::sqrt(ss / d + eps)", "std::sqrt(ss / (d - 1) + eps)"),
    ("Eq. 5: one slot short", "for (int j = 0; j < kf; ++j) count[order[j]]++;",
     "for (int j = 0; j + 1 < kf; ++j) count[order[j]]++;"),
    ("Eq. 37: a transfer on the same server", "        if (s != m) {\n          double trans",
     "        if (true) {\n          double trans"),
    ("Eq. 36: location taken from the home server", "const int s = loc[t];", "const int s = home[t];"),
    ("Eq. 44: the token's loss restarts at 0", "float q = qhat[t];", "float q = 0.0f;"),
    ("Eq. 44: loss not written back", "    qhat[t] = q;\n", "\n"),
    ("Eq. 42: minimum started at 0", "    if (p == 0.0f) continue;\n    float best = INFINITY;",
     "    if (p == 0.0f) continue;\n    float best = 0.0f;"),
    ("Eq. 43: horizon one short",
     "cost = cost + orc_phi(H - 1, tabs.data(), P, E, M, a, m, kk, qn, qbar);",
     "cost = cost + orc_phi(H - 2, tabs.data(), P, E, M, a, m, kk, qn, qbar);"),
    ("Eq. 42: deeper levels get the loss from before the substitute",
     "orc_phi(h - 1, tabs + 1, P + (size_t)E * E, E, M, a, m2, kk, q2, qbar)",
     "orc_phi(h - 1, tabs + 1, P + (size_t)E * E, E, M, a, m2, kk, qacc, qbar)"),
    ("Eq. 13: transfer time z * B", "double trans = z / B[s * M + m] + tau[s * M + m];",
     "double trans = z * B[s * M + m] + tau[s * M + m];"),
    ("Eq. 27: the expert left out of its group's mean",
     "if (group[k] == group[j]) { s += sim[j * E + k]; ++size; }",
     "if (group[k] == group[j] && k != j) { s += sim[j * E + k]; ++size; }"),
    ("Eq. 42: deeper levels measured from the home server",
     "orc_phi(h - 1, tabs + 1, P + (size_t)E * E, E, M, a, m2, kk, q2, qbar)",
     "orc_phi(h - 1, tabs + 1, P + (size_t)E * E, E, M, a, a, kk, q2, qbar)"),
    ("Eq. 42: deeper levels follow the target, not the executed expert",
     "orc_phi(h - 1, tabs + 1, P + (size_t)E * E, E, M, a, m2, kk, q2, qbar)",
     "orc_phi(h - 1, tabs + 1, P + (size_t)E * E, E, M, a, m2, kt, q2, qbar)"),
    ("Eq. 42: any substitute of the next target", "if (!((t1.subst[kt] >> kk) & 1u)) continue;", ""),
    ("Eq. 42: any server for the next expert", "if (!((t1.pmask[kk] >> m2) & 1u)) continue;", ""),
    ("Eq. 43: cost-to-go from the pre-layer location",
     "cost = cost + orc_phi(H - 1, tabs.data(), P, E, M, a, m, kk, qn, qbar);",
     "cost = cost + orc_phi(H - 1, tabs.data(), P, E, M, a, s, kk, qn, qbar);"),
    ("Eq. 32: coverage updated on server 0",
     "    y[((size_t)bm * L + bl) * E + group[bl * E + bj]] = 1;",
     "    y[((size_t)0 * L + bl) * E + group[bl * E + bj]] = 1;"),
    ("Eq. 35: memory charged to server 0", "used[bm] += p[bl * E + bj];", "used[0] += p[bl * E + bj];"),
    ("Eq. 34: replica not written", "placement[((size_t)bl * M + bm) * E + bj] = 1;", ""),
    ("Eq. 32: initial coverage from server 0's placement",
     "if (placement[((size_t)l * M + m) * E + j])\n          y[",
     "if (placement[((size_t)l * M + 0) * E + j])\n          y["),
] + [
    # the same rules in the look-ahead's own copy of the selection loop
    ("look-ahead tie: substitute before the exact expert", LA_TIE,
     LA_TIE.replace("better = sub < best_sub;", "better = sub > best_sub;")),
    ("look-ahead Eq. 44: loss not accumulated", LA_END,
     LA_END.replace("        q = q + Qtab[r * E + best_k];\n", "")),
    ("look-ahead Eq. 44: location from the last slot", LA_END,
     LA_END.replace("if (j == 0) first_server = best_m;", "first_server = best_m;")),
    ("look-ahead: distinct experts ignored", LA_DIST,
     LA_DIST.replace("          if ((taken >> kk) & 1u) continue;\n", "")),
]


CONFTEST = """
import pytest


@pytest.fixture(scope="session")
def orc():
    import oracle
    if "mutant" not in oracle.__file__:  # rc 3, never the rc 1 of a caught mistake
        pytest.exit("the real oracle was imported: " + oracle.__file__, returncode=3)
    oracle.lib()
    return oracle
"""


def run_mutant(orig, bad, base):
    """Builds the oracle with one planted mistake under `base` and runs the pins
    against it; returns the pytest process result."""
    src = open(SRC).read()
    # an anchor that occurs more than once is mutated at its first occurrence
    assert src.count(orig) >= 1, "mutation anchor not found: %r" % orig
    pkg = base / "oracle"
    pkg.mkdir(parents=True)
    for f in ("__init__.py", "build.py"):
        shutil.copy(os.path.join(ROOT, "oracle", f), pkg / f)
    (pkg / "ordermoe_oracle.cpp").write_text(src.replace(orig, bad, 1))
    subprocess.run([sys.executable, str(pkg / "build.py")], check=True, capture_output=True)
    tdir = base / "pins"
    tdir.mkdir()
    shutil.copy(os.path.join(ROOT, "tests", "test_oracle_pins.py"), tdir / "test_oracle_pins.py")
    (tdir / "conftest.py").write_text(CONFTEST)
    env = dict(os.environ, PYTHONPATH=str(base) + os.pathsep + ROOT, OMP_NUM_THREADS="1")
    return subprocess.run([sys.executable, "-m", "pytest", str(tdir), "-q", "-x", "-p", "no:cacheprovider",
                           "--rootdir", str(base)],
                          capture_output=True, text=True, env=env, cwd=str(base))


@pytest.fixture(scope="session")
def mutant_results(tmp_path_factory):
    """Every mutant built and checked once, side by side on the host cores."""
    from concurrent.futures import ThreadPoolExecutor
    root = tmp_path_factory.mktemp("mutants")
    workers = max(1, min(len(MUTANTS), os.cpu_count() or 1))
    with ThreadPoolExecutor(max_workers=workers) as ex:
        futs = {name: ex.submit(run_mutant, orig, bad, root / ("m%02d" % i))
                for i, (name, orig, bad) in enumerate(MUTANTS)}
        return {name: f.result() for name, f in futs.items()}


@pytest.mark.parametrize("name,orig,bad", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_planted_mistake(name, orig, bad, mutant_results):
    r = mutant_results[name]
    assert r.returncode == 1, "no pin caught the planted mistake %r (rc %d):\n%s" % (
        name, r.returncode, r.stdout[-2000:])
