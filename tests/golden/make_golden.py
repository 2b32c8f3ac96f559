"""Writes the golden fixtures of this directory from the oracle alone.

The paper prints no numeric worked example, so these fixtures pin the oracle
to itself over time: small seeded cases, their inputs and the oracle's outputs,
each citing the equations it exercises. tests/test_oracle_golden.py recomputes
them and requires exact equality; a deliberate change to the oracle's
arithmetic regenerates them with this script (python tests/golden/make_golden.py)
and names, in its commit, the passage that justifies it.
"""
import json
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(os.path.dirname(HERE)))

import oracle  # noqa: E402


def params(M, seed):
    rng = np.random.default_rng(seed)
    F = rng.uniform(20e12, 110e12, M)
    B = rng.uniform(1e8, 1.25e9, (M, M))
    tau = rng.uniform(2e-4, 2e-2, (M, M))
    np.fill_diagonal(tau, 0.0)
    return F, B, tau


def case_selection():
    """Eqs. 7, 18, 37-40, 43-44: tables and one layer's selection."""
    rng = np.random.default_rng(101)
    E, M, k, T = 6, 3, 2, 24
    W = rng.standard_normal((E, 5)); W[:, 0] += 2.0 * (np.arange(E) % 2)
    W /= np.linalg.norm(W, axis=1, keepdims=True)
    sim = (W @ W.T).astype(np.float32); np.fill_diagonal(sim, 1.0)
    group = (np.arange(E) % 2).astype(np.int32)
    x = np.zeros((M, E), np.uint8); x[np.arange(E) % M, np.arange(E)] = 1; x[0, 3] = 1
    F, B, tau = params(M, 102)
    z, c, theta, qbar = 8192.0, 3.5e8, 0.3, 0.25
    tab = oracle.tables(sim, group, x, theta, qbar, F, B, tau, z, c, 0.5, 0.5)
    logits = rng.standard_normal((T, E)).astype(np.float32)
    idx, w = oracle.topk(logits, k)
    home = rng.integers(0, M, T).astype(np.uint8)
    loc = np.where(rng.random(T) < 0.5, home, rng.integers(0, M, T)).astype(np.uint8)
    qhat = (rng.random(T) * 0.1).astype(np.float32)
    ch, sv, kd, loc2, q2 = oracle.select(idx, tab, home, loc, qhat)
    return {
        "cite": "Section III-B/C/E and V-B: Eqs. 7, 18, 37-40, 43-44 (Alg. 2, H = 1)",
        "inputs": {"sim": sim, "group": group, "placement": x, "F": F, "B": B, "tau": tau, "z": z,
                   "c": c, "theta": theta, "qbar": qbar, "logits": logits, "home": home,
                   "loc": loc, "qhat": qhat, "k": k},
        "outputs": {"Qtab": tab.Qtab, "Cq": tab.Cq, "A": tab.A, "topk_idx": idx, "topk_w": w,
                    "chosen": ch, "server": sv, "kind": kd, "loc": loc2, "qhat": q2},
    }


def case_plan():
    """Eqs. 4-6, 24-35: similarity, grouping, importance, placement, redundancy."""
    rng = np.random.default_rng(201)
    L, E, M, N, d, kf = 3, 8, 4, 64, 16, 2
    Wr = rng.standard_normal((L, E, d)).astype(np.float32)
    Wr[:, :, 0] += 3.0 * (np.arange(E) // 4)[None, :]
    X = rng.standard_normal((N, d)).astype(np.float32)
    bits = lambda a: (np.ascontiguousarray(a, np.float32).view(np.uint32) >> 16).astype(np.uint16)
    sims, counts, groups, imps, thetas = [], [], [], [], []
    for l in range(L):
        s, H = oracle.similarity(bits(Wr[l]), bits(X), return_H=True)
        cnt = oracle.expert_counts(np.ascontiguousarray(H.T), kf)
        th = oracle.theta(l + 1, L, 0.5, 0.9, 0.5)
        g, K, _ = oracle.group(s, cnt, th)
        sims.append(s); counts.append(cnt); groups.append(g); thetas.append(th)
        imps.append(oracle.importance(s, cnt, g))
    p = rng.integers(1, 3, (L, E)).astype(np.float64)
    C = np.array([9.0, 7.0, 6.0, 8.0]) * 2.0
    x, used, rc = oracle.place(np.stack(groups), np.stack(imps), p, C)
    pi = np.array([0.4, 0.3, 0.2, 0.1])
    x2, used2, reps = oracle.replicate(np.stack(groups), np.stack(imps), p, C, pi, x, used)
    return {
        "cite": "Section IV: Eqs. 4-6, 24-35 (Alg. 1)",
        "inputs": {"W_r_bf16": bits(Wr), "X_bf16": bits(X), "k_freq": kf, "p": p, "C": C, "pi": pi},
        "outputs": {"sim": np.stack(sims), "counts": np.stack(counts), "theta": np.array(thetas),
                    "group": np.stack(groups), "importance": np.stack(imps), "placement": x,
                    "used": used, "status": rc, "placement_redundant": x2, "used_redundant": used2,
                    "replicas": reps},
    }


def case_lookahead_and_cost():
    """Eqs. 13-23, 41-45: transitions, look-ahead selection, edge cost, utility."""
    rng = np.random.default_rng(301)
    L, E, M, k, T, H = 3, 6, 3, 2, 16, 3
    F, B, tau = params(M, 302)
    tabs, Qtabs = [], []
    for l in range(L):
        W = rng.standard_normal((E, 4)); W /= np.linalg.norm(W, axis=1, keepdims=True)
        sim = (W @ W.T).astype(np.float32); np.fill_diagonal(sim, 1.0)
        group = (np.arange(E) % 2).astype(np.int32)
        x = (rng.random((M, E)) < 0.5).astype(np.uint8); x[np.arange(E) % M, np.arange(E)] = 1
        t = oracle.tables(sim, group, x, 0.2, 0.3, F, B, tau, 8192.0, 3.5e8, 0.5, 0.5)
        tabs.append(t); Qtabs.append(t.Qtab)
    cal = rng.standard_normal((200, L, E)).astype(np.float32)
    tcnt, P = oracle.transitions(cal, k)
    home = rng.integers(0, M, T).astype(np.uint8)
    loc, q = home.copy(), np.zeros(T, np.float32)
    rec_t, rec_c, rec_s = [], [], []
    for l in range(L):
        logits = rng.standard_normal((T, E)).astype(np.float32)
        idx, _ = oracle.topk(logits, k)
        Hl = min(H, L - l)
        ch, sv, kd, loc, q = oracle.select_lookahead(idx, tabs[l:l + Hl], P[l:l + Hl - 1], home, loc, q)
        rec_t.append(idx); rec_c.append(ch); rec_s.append(sv)
    d, ql, n = oracle.trajectory_cost(np.stack(rec_t), np.stack(rec_c), np.stack(rec_s), home, F, B,
                                      tau, 8192.0, 3.5e8, np.stack(Qtabs))
    util = oracle.utility(d, d * 1.25, ql, 0.3, 0.5, 0.5, 0.1)
    return {
        "cite": "Sections III-D/E/F and V-C/D: Eqs. 13-23, 41-45",
        "inputs": {"seed": 301, "calibration": cal, "home": home},
        "outputs": {"transition_counts": tcnt, "P": P, "chosen": np.stack(rec_c),
                    "server": np.stack(rec_s), "loc": loc, "qhat": q, "delay": d, "loss": ql,
                    "moves": n, "utility": np.array(util)},
    }


def encode(v):
    """Arrays as {dtype, shape, hex of the little-endian bytes}: exact and compact."""
    if isinstance(v, np.ndarray):
        a = np.ascontiguousarray(v)
        return {"dtype": a.dtype.str, "shape": list(a.shape), "hex": a.tobytes().hex()}
    if isinstance(v, (np.integer,)):
        return int(v)
    if isinstance(v, (np.floating,)):
        return float(v)
    return v


CASES = {"selection_one_layer": case_selection, "plan_three_layers": case_plan,
         "lookahead_and_edge_cost": case_lookahead_and_cost}


def main():
    for name, fn in CASES.items():
        case = fn()
        out = {"case": name, "cite": case["cite"],
               "inputs": {k: encode(v) for k, v in case["inputs"].items()},
               "outputs": {k: encode(v) for k, v in case["outputs"].items()}}
        with open(os.path.join(HERE, name + ".json"), "w") as f:
            json.dump(out, f, indent=1)
        print("wrote", name)


if __name__ == "__main__":
    main()
