"""Pins for the CPU oracle: each check ties an oracle function to something
other than itself (exact arithmetic, a library routine on a special case, a
closed form, an invariant the paper states, or brute-force enumeration on a
tiny input), chosen so that a dropped term, a wrong sign or index, or a
transposed operand fails at least one of them.
"""
import itertools
from fractions import Fraction

import numpy as np
import pytest
import scipy.special
import torch
from scipy.spatial.distance import cdist

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def bf16_bits(a):
    """float array -> bf16 bit patterns (torch's round-to-nearest-even)."""
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def bits_to_f(b):
    return (np.asarray(b, np.uint16).astype(np.uint32) << 16).view(np.float32)


def rnd_bf16(rng, shape, std=1.0):
    return bf16_bits(rng.standard_normal(shape) * std)


# --------------------------------------------------------------------------
# Router logits (Eq. 3 per token)

def test_router_logits_exact_rational(orc):
    rng = np.random.default_rng(1)
    X = rnd_bf16(rng, (5, 7)); W = rnd_bf16(rng, (3, 7))
    got = orc.router_logits(X, W)
    xf, wf = bits_to_f(X), bits_to_f(W)
    for t in range(5):
        for e in range(3):
            exact = sum(Fraction(float(xf[t, c])) * Fraction(float(wf[e, c])) for c in range(7))
            assert got[t, e] == np.float32(float(exact))


def test_sums_are_exact_before_their_one_rounding(orc):
    """The oracle's sums (the router logits and the similarity's H, Eq. 3;
    the weighted combine of a token's slots) are exact up to their single
    final rounding: 2^24 + 1 - 2^24 is 1, although a running fp32 sum would
    lose the 1 to rounding. All inputs are exact in bf16."""
    big = 2.0 ** 12
    # router: x . w = 2^24 + 1 - 2^24
    X = bf16_bits([[big, 1.0, big]]); W = bf16_bits([[big, 1.0, -big]])
    assert orc.router_logits(X, W)[0, 0] == 1.0
    # combine: sum_j w_j Y_j with Y = (2^24, 1, -2^24) and unit weights
    Y = bf16_bits([[2.0 ** 24], [1.0], [-(2.0 ** 24)]])
    y = orc.combine(Y, np.array([[0, 1, 2]], np.int32), np.ones((1, 3), np.float32))
    assert bits_to_f(y)[0, 0] == 1.0
    # similarity: expert 0's activations are (1, 1) only when the cancelling
    # token keeps its 1; expert 1's are (2^12, 0): Sim = 1 / sqrt(2)
    Wr = bf16_bits([[big, 1.0, -big], [1.0, 0.0, 0.0]])
    Xc = bf16_bits([[big, 1.0, big], [0.0, 1.0, 0.0]])
    sim, H = orc.similarity(Wr, Xc, return_H=True)
    np.testing.assert_array_equal(H, np.array([[1.0, 1.0], [big, 0.0]], np.float32))
    assert sim[0, 1] == np.float32(1.0 / np.sqrt(2.0))


def test_router_logits_one_hot_tokens_pick_weight_columns(orc):
    rng = np.random.default_rng(2)
    E, d = 3, 11
    W = rnd_bf16(rng, (E, d))
    cols = np.array([0, 4, 10, 7])
    X = np.zeros((4, d), np.float32); X[np.arange(4), cols] = 1.0
    got = orc.router_logits(bf16_bits(X), W)
    np.testing.assert_array_equal(got, bits_to_f(W)[:, cols].T)


# --------------------------------------------------------------------------
# Softmax + top-k

def brute_topk(l, k):
    E = len(l)
    rank = [sum(1 for f in range(E) if l[f] > l[e] or (l[f] == l[e] and f < e)) for e in range(E)]
    return [rank.index(j) for j in range(k)]


def test_topk_brute_force_and_library_softmax(orc):
    rng = np.random.default_rng(3)
    for E, k in [(4, 1), (6, 2), (8, 3), (5, 5)]:
        logits = rng.standard_normal((20, E)).astype(np.float32)
        logits[0, :] = 0.5          # all tied
        logits[1, 1] = logits[1, 3]  # a tie inside
        for renorm in (0, 1):
            idx, w = orc.topk(logits, k, renorm)
            p = scipy.special.softmax(logits.astype(np.float64), axis=1)
            for t in range(20):
                sel = brute_topk(list(logits[t]), k)
                assert list(idx[t]) == sel
                ref = p[t, sel] / (p[t, sel].sum() if renorm else 1.0)
                np.testing.assert_allclose(w[t], ref, rtol=1e-6)


def test_topk_nan_is_an_error(orc):
    logits = np.zeros((2, 4), np.float32); logits[1, 2] = np.nan
    with pytest.raises(orc.OracleError):
        orc.topk(logits, 2)


# --------------------------------------------------------------------------
# Tables (Eqs. 7, 18, 37, 38)

def _params(rng, M):
    F = rng.uniform(20e12, 110e12, M)
    B = rng.uniform(1e9, 1e10, (M, M)); B = (B + B.T) / 2
    tau = rng.uniform(2e-4, 2e-2, (M, M)); tau = (tau + tau.T) / 2
    return F, B, tau


def test_tables_delay_term_closed_forms(orc):
    rng = np.random.default_rng(4)
    M, E = 4, 3
    F, B, tau = _params(rng, M)
    sim = np.eye(E, dtype=np.float32); group = np.arange(E, dtype=np.int32)
    x = np.ones((M, E), np.uint8)
    z, c, wT = 8192.0, 3.5e8, 0.5
    tab = orc.tables(sim, group, x, 0.5, 0.1, F, B, tau, z, c, wT, 0.5)
    A = tab.A.astype(np.float64)
    for a in range(M):
        # home server, no move: the delay equals d_ref, so the term is omega_T
        assert tab.A[a, a, a] == np.float32(wT)
        for s in range(M):
            # staying on s: omega_T * F_a / F_s (Eq. 37 with no transfer)
            np.testing.assert_allclose(A[a, s, s], wT * F[a] / F[s], rtol=1e-6)
            for m in range(M):
                if m == s:
                    continue
                # moving s -> m costs omega_T * F_a / c * (z / B_sm + tau_sm) extra
                extra = wT * F[a] / c * (z / B[s, m] + tau[s, m])
                np.testing.assert_allclose(A[a, s, m] - A[a, m, m], extra, rtol=1e-5)
    # no transfer cost at all: the term depends on the executing server only
    tab0 = orc.tables(sim, group, x, 0.5, 0.1, F, B, tau * 0, 0.0, c, wT, 0.5)
    for a, s, m in itertools.product(range(M), repeat=3):
        np.testing.assert_allclose(tab0.A[a, s, m], wT * F[a] / F[m], rtol=1e-6)


def test_tables_quality_terms_closed_forms(orc):
    E = 4
    sim = np.array([[1.0, 0.5, -1.0, 0.75],
                    [0.5, 1.0, 0.0, 1.25],   # 1.25: rounding overshoot, clamps to zero loss
                    [-1.0, 0.0, 1.0, 0.5],
                    [0.75, 1.25, 0.5, 1.0]], np.float32)
    group = np.array([0, 0, 1, 0], np.int32)
    x = np.ones((2, E), np.uint8)
    F = np.array([1e13, 2e13]); B = np.ones((2, 2)) * 1e9; tau = np.zeros((2, 2))
    tab = orc.tables(sim, group, x, 0.6, 0.25, F, B, tau, 1.0, 1.0, 0.5, 0.5)
    expect_Q = np.array([[0, 0.25, 1.0, 0.125],
                         [0.25, 0, 0.5, 0.0],
                         [1.0, 0.5, 0, 0.25],
                         [0.125, 0.0, 0.25, 0]], np.float32)
    np.testing.assert_array_equal(tab.Qtab, expect_Q)
    # Cq = omega_Q * Q / Qbar = 0.5 * Q / 0.25 = 2 Q
    np.testing.assert_array_equal(tab.Cq, 2 * expect_Q)
    # R_{l,r}: same group, k != r, Sim >= 0.6
    subst = [int(v) for v in tab.subst]
    assert subst[0] == (1 << 3)              # 1: Sim 0.5 < 0.6; 3: 0.75
    assert subst[1] == (1 << 3)              # 3: Sim 1.25 >= 0.6
    assert subst[2] == 0                     # alone in group 1
    assert subst[3] == (1 << 0) | (1 << 1)
    # Eq. 7's threshold is inclusive: a similarity equal to theta qualifies
    tab2 = orc.tables(sim, group, x, 0.75, 0.25, F, B, tau, 1.0, 1.0, 0.5, 0.5)
    assert int(tab2.subst[0]) == (1 << 3)    # Sim(0, 3) = 0.75 = theta
    assert int(tab2.subst[3]) == (1 << 0) | (1 << 1)


def test_tables_placement_mask(orc):
    E, M = 5, 3
    x = np.zeros((M, E), np.uint8); x[0, 0] = x[2, 0] = x[1, 3] = x[2, 4] = x[0, 1] = x[1, 2] = 1
    F = np.ones(M) * 1e13; B = np.ones((M, M)) * 1e9; tau = np.zeros((M, M))
    tab = orc.tables(np.eye(E, dtype=np.float32), np.arange(E, dtype=np.int32), x, 0.5, 0.1,
                     F, B, tau, 1.0, 1.0, 0.5, 0.5)
    assert [int(v) for v in tab.pmask] == [0b101, 0b001, 0b010, 0b010, 0b100]


# --------------------------------------------------------------------------
# Selection (Alg. 2, H = 1) against brute-force enumeration of every
# (server, expert) pair, following Eqs. 7, 8, 18, 37, 38, 40, 43, 44.

def brute_select(idx, sim, group, x, theta, qbar, F, B, tau, z, c, wT, wQ, home, loc, qhat):
    T, k = idx.shape
    M, E = x.shape
    f32 = np.float32
    chosen = np.zeros((T, k), np.int32); server = np.zeros((T, k), np.uint8)
    kind = np.zeros((T, k), np.uint8)
    loc2 = loc.copy(); q2 = qhat.copy()

    def quality(r, kk):  # Eq. 18, phi = identity, fp32
        if kk == r:
            return f32(0)
        return f32(f32(0.5) * (f32(1) - min(f32(sim[r, kk]), f32(1))))

    def delay_term(a, s, m):  # Eqs. 37-38 delay term, fp64 -> fp32
        dl = c / F[m] if s == m else (z / B[s, m] + tau[s, m]) + c / F[m]
        return f32(wT * dl / (c / F[a]))

    for t in range(T):
        a, s, q = int(home[t]), int(loc[t]), f32(qhat[t])
        used = set(int(v) for v in idx[t])
        for j in range(k):
            r = int(idx[t, j])
            cands = []
            for m in range(M):
                for kk in range(E):
                    if not x[m, kk]:
                        continue
                    if kk != r:
                        if group[kk] != group[r] or not (sim[r, kk] >= f32(theta)):
                            continue
                        if kk in used:
                            continue
                        if not (f32(q + quality(r, kk)) <= f32(qbar)):
                            continue
                    Q = quality(r, kk)
                    qterm = f32(0) if Q == 0 else f32(wQ * float(Q) / float(f32(qbar)))
                    cost = f32(delay_term(a, s, m) + (f32(0) if kk == r else qterm))
                    cands.append((cost, kk != r, m != s, m, kk))
            best = min(cands)
            _, sub, away, m, kk = best
            chosen[t, j] = kk; server[t, j] = m; kind[t, j] = 2 * away + sub
            if sub:
                used.add(kk)
                q = f32(q + quality(r, kk))
            if j == 0:
                loc2[t] = m
        q2[t] = q
    return chosen, server, kind, loc2, q2


def random_case(rng, E, M, k, T, kgroups):
    Wt = rng.standard_normal((E, 5))
    Wt[:, 0] += 3.0 * (np.arange(E) % kgroups)  # correlate same-group rows
    sim = (1 - cdist(Wt, Wt, "cosine")).astype(np.float32)
    np.fill_diagonal(sim, 1.0)
    group = (np.arange(E) % kgroups).astype(np.int32)
    x = (rng.random((M, E)) < 0.4).astype(np.uint8)
    for e in range(E):
        if not x[:, e].any():
            x[rng.integers(M), e] = 1
    F, B, tau = _params(rng, M)
    if rng.random() < 0.5:   # cheap links so that remote candidates compete
        tau = tau * 1e-4
    theta = float(rng.choice([-0.5, 0.0, 0.3, 0.6]))
    qbar = float(rng.choice([0.0, 0.1, 0.3, 1.0]))
    logits = rng.standard_normal((T, E)).astype(np.float32)
    idx = np.argsort(-logits, axis=1, kind="stable")[:, :k].astype(np.int32)
    home = rng.integers(0, M, T).astype(np.uint8)
    loc = np.where(rng.random(T) < 0.5, home, rng.integers(0, M, T)).astype(np.uint8)
    qhat = (rng.random(T) * qbar * 0.8).astype(np.float32)
    return dict(idx=idx, sim=sim, group=group, x=x, theta=theta, qbar=qbar, F=F, B=B, tau=tau,
                z=2048.0, c=1e9, wT=float(rng.choice([0.0, 0.3, 0.5])), wQ=0.5,
                home=home, loc=loc, qhat=qhat)


def run_oracle_select(orc, cs):
    tab = orc.tables(cs["sim"], cs["group"], cs["x"], cs["theta"], cs["qbar"], cs["F"], cs["B"],
                     cs["tau"], cs["z"], cs["c"], cs["wT"], cs["wQ"])
    return orc.select(cs["idx"], tab, cs["home"], cs["loc"], cs["qhat"]), tab


def test_select_matches_brute_force(orc):
    rng = np.random.default_rng(5)
    n = 0
    for trial in range(300):
        E = int(rng.integers(2, 7)); M = int(rng.integers(1, 4)); k = int(rng.integers(1, min(E, 3) + 1))
        cs = random_case(rng, E, M, k, 6, int(rng.integers(1, 3)))
        (ch, sv, kd, loc, q), _ = run_oracle_select(orc, cs)
        bch, bsv, bkd, bloc, bq = brute_select(**cs)
        np.testing.assert_array_equal(ch, bch)
        np.testing.assert_array_equal(sv, bsv)
        np.testing.assert_array_equal(kd, bkd)
        np.testing.assert_array_equal(loc, bloc)
        np.testing.assert_array_equal(q, bq)
        n += int((kd % 2 == 1).sum())
    assert n > 50   # substitutes were exercised


def test_select_invariants(orc):
    rng = np.random.default_rng(6)
    for trial in range(200):
        E = int(rng.integers(2, 9)); M = int(rng.integers(1, 5)); k = int(rng.integers(1, min(E, 4) + 1))
        cs = random_case(rng, E, M, k, 16, int(rng.integers(1, 4)))
        (ch, sv, kd, loc, q), tab = run_oracle_select(orc, cs)
        for t in range(16):
            assert len(set(ch[t])) == k                                  # k distinct experts
            for j in range(k):
                r, kk, m = cs["idx"][t, j], ch[t, j], sv[t, j]
                assert cs["x"][m, kk] == 1                               # c.6
                if kk != r:                                              # c.7 / Eq. 7
                    assert cs["group"][kk] == cs["group"][r]
                    assert cs["sim"][r, kk] >= np.float32(cs["theta"])
                assert (kd[t, j] & 1) == (kk != r)
                assert (kd[t, j] >> 1) == (m != cs["loc"][t])
            assert q[t] <= np.float32(cs["qbar"])                        # Property 2
            assert loc[t] == sv[t, 0]


def test_select_identity_when_every_expert_is_everywhere(orc):
    rng = np.random.default_rng(7)
    cs = random_case(rng, 6, 3, 2, 32, 2)
    cs["x"] = np.ones((3, 6), np.uint8)
    cs["qbar"] = 1.0; cs["theta"] = -1.0; cs["wT"] = 0.5
    cs["F"], cs["B"], cs["tau"] = _params(rng, 3)      # testbed links: >= 0.2 ms per move
    (ch, sv, kd, loc, q), _ = run_oracle_select(orc, cs)
    np.testing.assert_array_equal(ch, cs["idx"])
    assert (kd == 0).all() and (sv == cs["loc"][:, None]).all()
    assert (q == cs["qhat"]).all()


def test_select_no_budget_or_high_threshold_is_pure_exact(orc):
    rng = np.random.default_rng(8)
    for over in ({"qbar": 0.0}, {"theta": 1.5}):
        cs = random_case(rng, 6, 3, 2, 32, 2)
        cs["qhat"] = np.zeros(32, np.float32)
        cs.update(over)
        (ch, sv, kd, loc, q), _ = run_oracle_select(orc, cs)
        np.testing.assert_array_equal(ch, cs["idx"])
        assert (kd % 2 == 0).all()


def test_select_ties_prefer_current_then_lower_server(orc):
    E, M = 3, 3
    sim = np.eye(E, dtype=np.float32)
    x = np.zeros((M, E), np.uint8); x[1, 0] = x[2, 0] = 1; x[0, 1] = x[0, 2] = 1
    F = np.ones(M) * 1e13; B = np.ones((M, M)) * 1e9; tau = np.ones((M, M)) * 1e-3
    tab = orc.tables(sim, np.arange(E, dtype=np.int32), x, 0.5, 0.1, F, B, tau, 1.0, 1.0, 0.0, 0.5)
    idx = np.array([[0], [0]], np.int32)          # omega_T = 0: every exact costs 0
    ch, sv, kd, loc, q = orc.select(idx, tab, np.array([2, 0], np.uint8),
                                    np.array([2, 0], np.uint8), np.zeros(2, np.float32))
    assert list(sv[:, 0]) == [2, 1]               # stay on 2; else lowest server 1
    assert list(kd[:, 0]) == [0, 2]


def test_select_local_first_with_testbed_parameters(orc):
    """With the testbed's ranges (Section VI-A) every remote move costs more
    than any local candidate, so the choice is: keep the target if local, else
    the most similar feasible local substitute, else a remote candidate."""
    from paper_2607_17154_gb300 import synth
    rng = np.random.default_rng(9)
    E, M, k, d, dff = 8, 4, 2, 4096, 14336
    sp = synth.server_params(M, d, dff, seed=3)
    Wt = rng.standard_normal((E, 6)); Wt[:, 0] += 4 * (np.arange(E) // 4)
    sim = (1 - cdist(Wt, Wt, "cosine")).astype(np.float32); np.fill_diagonal(sim, 1)
    group = (np.arange(E) // 4).astype(np.int32)
    x = np.zeros((M, E), np.uint8)
    for e in range(E):
        x[e % M, e] = 1
    theta, qbar = 0.0, 0.4
    tab = orc.tables(sim, group, x, theta, qbar, sp.F, sp.B, sp.tau, sp.z, sp.c, 0.5, 0.5)
    T = 64
    idx = np.array([rng.permutation(E)[:k] for _ in range(T)], np.int32)
    home = rng.integers(0, M, T).astype(np.uint8)
    ch, sv, kd, loc, q = orc.select(idx, tab, home, home.copy(), np.zeros(T, np.float32))
    for t in range(T):
        s = home[t]; used = set(idx[t]); qq = np.float32(0)
        for j in range(k):
            r = idx[t, j]
            if x[s, r]:
                assert ch[t, j] == r and sv[t, j] == s
                continue
            local = [kk for kk in range(E) if x[s, kk] and kk != r and group[kk] == group[r]
                     and sim[r, kk] >= theta and kk not in used
                     and np.float32(qq + tab.Qtab[r, kk]) <= np.float32(qbar)]
            if local:
                best = max(local, key=lambda kk: (sim[r, kk], -kk))
                assert ch[t, j] == best and sv[t, j] == s
                used.add(best); qq = np.float32(qq + tab.Qtab[r, best])
            else:
                # no local candidate: the token moves (to the target, or to a
                # substitute on a server with a cheaper link)
                assert sv[t, j] != s
                if ch[t, j] != r:
                    used.add(ch[t, j]); qq = np.float32(qq + tab.Qtab[r, ch[t, j]])


# --------------------------------------------------------------------------
# Permutation

def test_dispatch_is_a_stable_counting_sort(orc):
    rng = np.random.default_rng(10)
    for T, k, E in [(1, 1, 1), (7, 2, 5), (100, 3, 8), (33, 6, 64)]:
        chosen = rng.integers(0, E, (T, k)).astype(np.int32)
        if E > 3:
            chosen[chosen == 2] = 1       # an expert with no rows
        off, row_token, row_of = orc.dispatch(chosen, E)
        order = np.argsort(chosen.ravel(), kind="stable")
        np.testing.assert_array_equal(row_token, order // k)
        np.testing.assert_array_equal(off, np.concatenate([[0], np.cumsum(np.bincount(chosen.ravel(), minlength=E))]))
        inv = np.empty(T * k, np.int64); inv[order] = np.arange(T * k)
        np.testing.assert_array_equal(row_of.ravel(), inv)
        assert sorted(row_of.ravel()) == list(range(T * k))      # bijection


def test_gather_rows(orc):
    rng = np.random.default_rng(11)
    X = rnd_bf16(rng, (9, 16)); rt = rng.integers(0, 9, 20).astype(np.int32)
    np.testing.assert_array_equal(orc.gather_rows(X, rt), X[rt])


# --------------------------------------------------------------------------
# SwiGLU FFN

def test_ffn_one_hot_reduces_to_silu(orc):
    """x = e_0, W1[:, 0] = a, W3[:, 0] = 1, W2 a selection matrix: the expert
    output is bf16(silu(a)) routed through W2's selection, so the gate, the
    up projection, their order and both matrix orientations are all pinned."""
    rng = np.random.default_rng(12)
    E, d, dff = 2, 6, 10
    a = rng.standard_normal((E, dff)) * 3
    W1 = np.zeros((E, dff, d)); W1[:, :, 0] = a
    W1[:, :, 1:] = rng.standard_normal((E, dff, d - 1))   # never multiplied (x_c = 0)
    W3 = np.zeros((E, dff, d)); W3[:, :, 0] = 1.0; W3[:, :, 2] = 5.0
    W2 = np.zeros((E, d, dff))
    perm = [rng.permutation(dff)[:d] for _ in range(E)]
    for e in range(E):
        W2[e, np.arange(d), perm[e]] = 1.0
    X = np.zeros((4, d)); X[:, 0] = 1.0
    rows_e = np.array([0, 1, 1, 0], np.int32)
    W1b, W3b, W2b = bf16_bits(W1), bf16_bits(W3), bf16_bits(W2)
    H, Y = orc.ffn_rows(bf16_bits(X), rows_e, W1b, W3b, W2b)
    ab = bits_to_f(W1b)[:, :, 0].astype(np.float64)
    silu = ab * scipy.special.expit(ab)
    for r, e in enumerate(rows_e):
        np.testing.assert_array_equal(H[r], bf16_bits(silu[e]))
        np.testing.assert_array_equal(Y[r], H[r][perm[e]])


def test_ffn_zero_input_and_power_of_two_scaling(orc):
    rng = np.random.default_rng(13)
    E, d, dff = 3, 8, 12
    W1, W3, W2 = (rnd_bf16(rng, s, 0.5) for s in [(E, dff, d), (E, dff, d), (E, d, dff)])
    X = rnd_bf16(rng, (5, d)); re = np.array([0, 1, 2, 2, 0], np.int32)
    H0, Y0 = orc.ffn_rows(np.zeros_like(X), re, W1, W3, W2)
    assert (H0 == 0).all() and (bits_to_f(Y0) == 0).all()
    H, Y = orc.ffn_rows(X, re, W1, W3, W2)
    H2, Y2 = orc.ffn_rows(X, re, W1, W3, bf16_bits(bits_to_f(W2) * 4.0))
    np.testing.assert_array_equal(H2, H)
    np.testing.assert_array_equal(bits_to_f(Y2), bits_to_f(Y) * 4.0)
    # swapping the gate and up matrices changes the output (silu is not symmetric)
    Hs, Ys = orc.ffn_rows(X, re, W3, W1, W2)
    assert not np.array_equal(Hs, H)


def test_ffn_row_uses_its_own_expert(orc):
    rng = np.random.default_rng(14)
    E, d, dff = 3, 8, 16
    W1, W3, W2 = (rnd_bf16(rng, s, 0.5) for s in [(E, dff, d), (E, dff, d), (E, d, dff)])
    X = rnd_bf16(rng, (1, d))
    outs = [orc.ffn_rows(X, np.array([e], np.int32), W1, W3, W2)[1] for e in range(E)]
    for e in range(E):
        # the same row through expert e equals the row through a model whose
        # only expert is e
        solo = orc.ffn_rows(X, np.array([0], np.int32), W1[e:e + 1], W3[e:e + 1], W2[e:e + 1])[1]
        np.testing.assert_array_equal(outs[e], solo)
    assert not np.array_equal(outs[0], outs[1])


# --------------------------------------------------------------------------
# Combine

def test_combine_special_cases(orc):
    rng = np.random.default_rng(15)
    T, d = 6, 10
    Y = rnd_bf16(rng, (T, d))
    rof = np.arange(T, dtype=np.int32)[:, None]
    np.testing.assert_array_equal(orc.combine(Y, rof, np.ones((T, 1), np.float32)), Y)
    # two slots, small-integer rows and dyadic weights: exact
    Yi = bf16_bits(rng.integers(-8, 8, (2 * T, d)).astype(np.float32))
    rof2 = np.stack([np.arange(T), T + (np.arange(T) + 1) % T], 1).astype(np.int32)
    w = np.tile(np.array([0.75, 0.25], np.float32), (T, 1))
    yf = bits_to_f(orc.combine(Yi, rof2, w))
    Yf = bits_to_f(Yi)
    np.testing.assert_array_equal(yf, 0.75 * Yf[rof2[:, 0]] + 0.25 * Yf[rof2[:, 1]])


# --------------------------------------------------------------------------
# Residual map between stacked layers: RMSNorm and the residual add

def test_rmsnorm_closed_forms(orc):
    d = 16
    h = np.zeros((4, d), np.float32)
    h[0] = 1.0                           # mean square 1: x = 1/sqrt(1 + eps) -> 1.0 in bf16
    h[1] = -3.0                          # mean square 9: -3/3 = -1
    h[2, :8] = 2.0                       # mean square 2: 2/sqrt(2) = sqrt(2)
    h[3, 0] = 4.0                        # one non-zero: 4/sqrt(16/16) = 4, rest 0
    x = bits_to_f(orc.rmsnorm(bf16_bits(h), eps=1e-6))
    np.testing.assert_array_equal(x[0], np.ones(d, np.float32))
    np.testing.assert_array_equal(x[1], -np.ones(d, np.float32))
    np.testing.assert_array_equal(x[2], np.r_[np.full(8, bits_to_f(bf16_bits([np.sqrt(2.0)]))[0]),
                                              np.zeros(8)].astype(np.float32))
    np.testing.assert_array_equal(x[3], np.r_[[4.0], np.zeros(d - 1)].astype(np.float32))


def test_rmsnorm_epsilon_in_the_root(orc):
    """eps sits inside the root: a zero row stays zero (0 / sqrt(eps)), and a
    constant row c gives c / sqrt(c^2 + eps): with c = 2^-8 and eps = 2^-16
    that is 2^-8 / sqrt(2^-15) = sqrt(2) / 2 (1 without eps)."""
    d = 8
    h = np.zeros((2, d), np.float32)
    h[1] = 2.0 ** -8
    x = bits_to_f(orc.rmsnorm(bf16_bits(h), eps=2.0 ** -16))
    np.testing.assert_array_equal(x[0], np.zeros(d, np.float32))
    np.testing.assert_array_equal(x[1], np.full(d, bits_to_f(bf16_bits([np.sqrt(0.5)]))[0]))


def test_rmsnorm_scale_invariant_and_unit_rms(orc):
    rng = np.random.default_rng(41)
    h = rnd_bf16(rng, (7, 40), std=3.0)
    x = orc.rmsnorm(h, eps=1e-30)
    # a power-of-two scaling of h changes nothing (exact in binary, eps negligible)
    np.testing.assert_array_equal(orc.rmsnorm(bf16_bits(bits_to_f(h) * 8.0), eps=1e-30), x)
    np.testing.assert_array_equal(orc.rmsnorm(bf16_bits(bits_to_f(h) * -0.25), eps=1e-30),
                                  bf16_bits(-bits_to_f(x)))
    # every row has unit root mean square up to the bf16 rounding of x
    ms = (bits_to_f(x).astype(np.float64) ** 2).mean(axis=1)
    np.testing.assert_allclose(ms, 1.0, rtol=2 * 2.0 ** -8)


def test_combine_residual_special_cases(orc):
    rng = np.random.default_rng(42)
    T, k, d = 5, 3, 12
    Y = rnd_bf16(rng, (T * k, d))
    rof = rng.permutation(T * k).astype(np.int32).reshape(T, k)
    w = rng.random((T, k)).astype(np.float32)
    h = rnd_bf16(rng, (T, d))
    # zero weights: the residual stream passes through unchanged
    np.testing.assert_array_equal(orc.combine_residual(Y, rof, np.zeros((T, k), np.float32), h), h)
    # a zero residual stream: the plain weighted combine
    np.testing.assert_array_equal(orc.combine_residual(Y, rof, w, np.zeros_like(h)),
                                  orc.combine(Y, rof, w))
    # small integers and dyadic weights: every sum is exact
    Yi = bf16_bits(rng.integers(-8, 8, (T * k, d)).astype(np.float32))
    hi = bf16_bits(rng.integers(-16, 16, (T, d)).astype(np.float32))
    wd = np.tile(np.array([0.5, 0.25, 0.125], np.float32), (T, 1))
    got = bits_to_f(orc.combine_residual(Yi, rof, wd, hi))
    Yf = bits_to_f(Yi)
    ref = bits_to_f(hi) + sum(wd[:, j:j + 1] * Yf[rof[:, j]] for j in range(k))
    np.testing.assert_array_equal(got, ref)


# --------------------------------------------------------------------------
# Similarity (Eqs. 3-4) and activation counts (Eq. 5)

def test_similarity_identity_calibration_is_cosine_of_router_rows(orc):
    rng = np.random.default_rng(16)
    E, d = 6, 12
    W = rnd_bf16(rng, (E, d))
    Wf = bits_to_f(W).astype(np.float64)
    sim = orc.similarity(W, bf16_bits(np.eye(d)))
    ref = 1 - cdist(Wf, Wf, "cosine")
    np.fill_diagonal(ref, 1.0)
    np.testing.assert_allclose(sim, ref, atol=1e-6)


def test_similarity_diagonal_calibration_scales_feature_columns(orc):
    rng = np.random.default_rng(17)
    E, d = 5, 9
    W = rnd_bf16(rng, (E, d)); s = np.array([1, 2, 0.5, 4, 1, 0.25, 8, 1, 2], np.float32)
    sim = orc.similarity(W, bf16_bits(np.diag(s)))
    Ws = bits_to_f(W).astype(np.float64) * s
    ref = 1 - cdist(Ws, Ws, "cosine"); np.fill_diagonal(ref, 1.0)
    np.testing.assert_allclose(sim, ref, atol=1e-6)


def test_similarity_invariants(orc):
    rng = np.random.default_rng(18)
    E, d, N = 7, 16, 40
    W = rnd_bf16(rng, (E, d)); Xc = rnd_bf16(rng, (N, d))
    Wf = bits_to_f(W).copy()
    Wf[3] = Wf[1]              # identical rows
    Wf[5] = -2 * Wf[2]         # opposite direction
    Wf[6] = 0                  # a dead expert
    W = bf16_bits(Wf)
    sim = orc.similarity(W, Xc)
    np.testing.assert_array_equal(sim, sim.T)
    assert (np.diag(sim) == 1).all() and (np.abs(sim) <= 1 + 1e-6).all()
    assert sim[1, 3] == pytest.approx(1.0, abs=1e-6)
    assert sim[2, 5] == pytest.approx(-1.0, abs=1e-6)
    assert (sim[6, :6] == 0).all()
    Ws = Wf.copy(); Ws[0] *= 4
    np.testing.assert_allclose(orc.similarity(bf16_bits(Ws), Xc), sim, atol=1e-6)
    # duplicating every calibration token leaves the cosine unchanged
    np.testing.assert_allclose(orc.similarity(W, np.concatenate([Xc, Xc])), sim, atol=1e-6)


def test_expert_counts_brute_force(orc):
    rng = np.random.default_rng(19)
    logits = rng.standard_normal((50, 6)).astype(np.float32)
    logits[3] = 1.0
    for kf in (1, 2, 6):
        cnt = orc.expert_counts(logits, kf)
        ref = np.zeros(6, np.int64)
        for t in range(50):
            for e in brute_topk(list(logits[t]), kf):
                ref[e] += 1
        np.testing.assert_array_equal(cnt, ref)
        assert cnt.sum() == 50 * kf


# --------------------------------------------------------------------------
# Threshold, grouping, importance, placement (Eqs. 6, 24-31)

def test_theta_endpoints_and_monotone(orc):
    N = 24
    th = [float(orc.theta(l, N, 0.5, 0.9, 0.7)) for l in range(1, N + 1)]
    assert th[0] == pytest.approx(0.9) and th[-1] == pytest.approx(0.5)
    assert all(a > b for a, b in zip(th, th[1:]))
    assert float(orc.theta(1, 1, 0.5, 0.9, 0.7)) == pytest.approx(0.7)
    assert th[11] == pytest.approx(0.5 + 0.4 * 12 / 23, abs=1e-7)


def hand_tables(orc, E, M, qbar, A, Q=None, Cq=None, subst=None, pmask=None):
    """Selection tables written by hand (dyadic values, so that sums and ties
    are exact in fp32): A[a][s][m], Qtab/Cq [E][E], subst bit masks, pmask."""
    Q = np.zeros((E, E), np.float32) if Q is None else np.asarray(Q, np.float32)
    Cq = np.zeros((E, E), np.float32) if Cq is None else np.asarray(Cq, np.float32)
    subst = np.zeros(E, np.uint64) if subst is None else np.asarray(subst, np.uint64)
    return orc.Tables(np.ascontiguousarray(Q), np.ascontiguousarray(Cq), np.ascontiguousarray(subst),
                      np.ascontiguousarray(np.asarray(A, np.float32)),
                      np.ascontiguousarray(np.asarray(pmask, np.uint32)), qbar, E, M)


def test_select_budget_is_inclusive(orc):
    """Eq. 40 admits a substitute when Q_hat + Q <= Qbar: at equality it is
    feasible. Target 0 sits only on remote server 1 (cost 1); substitute 1 on
    local server 0 costs Cq = 0.125 and brings the loss from 0.25 to exactly
    Qbar = 0.5."""
    E, M = 2, 2
    A = np.zeros((M, M, M), np.float32); A[0, 0, 1] = 1.0
    Q = [[0, 0.25], [0.25, 0]]; Cq = [[0, 0.125], [0.125, 0]]
    tab = hand_tables(orc, E, M, 0.5, A, Q, Cq, subst=[0b10, 0b01], pmask=[0b10, 0b01])
    ch, sv, kd, loc, q = orc.select(np.array([[0]], np.int32), tab, np.zeros(1, np.uint8),
                                    np.zeros(1, np.uint8), np.array([0.25], np.float32))
    assert (ch[0, 0], sv[0, 0], kd[0, 0]) == (1, 0, 1)
    assert q[0] == np.float32(0.5)


def test_select_equal_costs_prefer_the_exact_expert_then_the_lower_substitute(orc):
    """Ties of Eq. 43's cost: the exact target before a substitute (reading
    of the tie rule: sub < ...), and among equally cheap substitutes on the same
    server the lower expert index. Costs are dyadic, so the ties are exact."""
    E, M = 3, 2
    # exact target 0 on remote server 1 at 0.5; substitute 1 on local server 0 at 0.25 + Cq 0.25
    A = np.zeros((M, M, M), np.float32); A[0, 0, 1] = 0.5
    Cq = np.zeros((E, E), np.float32); Cq[0, 1] = 0.25
    Q = np.zeros((E, E), np.float32); Q[0, 1] = 0.125
    A[0, 0, 0] = 0.25
    tab = hand_tables(orc, E, M, 0.5, A, Q, Cq, subst=[0b010, 0, 0], pmask=[0b10, 0b01, 0b00])
    ch, sv, kd, _, _ = orc.select(np.array([[0]], np.int32), tab, np.zeros(1, np.uint8),
                                  np.zeros(1, np.uint8), np.zeros(1, np.float32))
    assert (ch[0, 0], sv[0, 0], kd[0, 0]) == (0, 1, 2)     # exact, remote: cost 0.5 either way
    # two substitutes 1 and 2 of target 0 on server 0 at the same cost; the target costs more
    A2 = np.zeros((M, M, M), np.float32); A2[0, 0, 1] = 1.0
    Cq2 = np.zeros((E, E), np.float32); Cq2[0, 1] = Cq2[0, 2] = 0.25
    Q2 = np.zeros((E, E), np.float32); Q2[0, 1] = Q2[0, 2] = 0.125
    tab2 = hand_tables(orc, E, M, 0.5, A2, Q2, Cq2, subst=[0b110, 0, 0],
                       pmask=[0b10, 0b01, 0b01])
    ch, sv, kd, _, _ = orc.select(np.array([[0]], np.int32), tab2, np.zeros(1, np.uint8),
                                  np.zeros(1, np.uint8), np.zeros(1, np.float32))
    assert (ch[0, 0], sv[0, 0], kd[0, 0]) == (1, 0, 1)


def test_lookahead_ties_follow_the_myopic_rule(orc):
    """With P = 0 the cost-to-go is 0 (every term has P = 0), so Eq. 43 with
    H = 2 takes the same decisions as H = 1, ties included: the exact target
    before an equally cheap substitute, and the lower of two equally cheap
    substitutes on one server."""
    E, M = 3, 2
    A = np.zeros((M, M, M), np.float32); A[0, 0, 1] = 0.5; A[0, 0, 0] = 0.25
    Cq = np.zeros((E, E), np.float32); Cq[0, 1] = 0.25
    Q = np.zeros((E, E), np.float32); Q[0, 1] = 0.125
    tab = hand_tables(orc, E, M, 0.5, A, Q, Cq, subst=[0b010, 0, 0], pmask=[0b10, 0b01, 0b00])
    A2 = np.zeros((M, M, M), np.float32); A2[0, 0, 1] = 1.0
    Cq2 = np.zeros((E, E), np.float32); Cq2[0, 1] = Cq2[0, 2] = 0.25
    Q2 = np.zeros((E, E), np.float32); Q2[0, 1] = Q2[0, 2] = 0.125
    tab2 = hand_tables(orc, E, M, 0.5, A2, Q2, Cq2, subst=[0b110, 0, 0], pmask=[0b10, 0b01, 0b01])
    P = np.zeros((1, E, E), np.float32)
    z = lambda: (np.zeros(1, np.uint8), np.zeros(1, np.uint8), np.zeros(1, np.float32))
    for t, want in ((tab, (0, 1, 2)), (tab2, (1, 0, 1))):
        ch, sv, kd, _, _ = orc.select_lookahead(np.array([[0]], np.int32), [t, t], P, *z())
        assert (ch[0, 0], sv[0, 0], kd[0, 0]) == want


def test_phi_budget_is_inclusive(orc):
    """Eq. 42 takes the next layer's substitutes under the same rule as Eq. 40:
    with Q_hat = 0.25 and Q(1 -> 0) = 0.25 the substitute is feasible at
    Q_hat + Q = Qbar = 0.5. From server 0 the next target 1 runs exactly on
    server 1 (cost 1) or as substitute 0 on server 0 (cost 0.125), with
    P(0 -> 1) = 1: Phi^(1) = 0.125."""
    E, M = 2, 2
    t0 = hand_tables(orc, E, M, 0.5, np.zeros((M, M, M), np.float32), pmask=[0b01, 0b01])
    A1 = np.zeros((M, M, M), np.float32); A1[0, 0, 1] = 1.0
    Q1 = [[0, 0.25], [0.25, 0]]; Cq1 = [[0, 0.125], [0.125, 0]]
    t1 = hand_tables(orc, E, M, 0.5, A1, Q1, Cq1, subst=[0b10, 0b01], pmask=[0b01, 0b10])
    P = np.array([[[0, 1], [1, 0]]], np.float32)
    assert orc.phi(1, [t0, t1], P, 0, 0, 0, 0.25) == 0.125
    assert orc.phi(1, [t0, t1], P, 0, 0, 0, 0.3) == 1.0     # above the budget: exact only


def test_phi_carries_a_substitute_loss_to_the_deeper_level(orc):
    """Eq. 42 with two future layers, Qbar = 0.5, Q_hat = 0.25. At layer l+1
    the next target 1 runs exactly on server 1 (cost 1) or as substitute 0 on
    server 0 (Cq 0.125), which brings the loss to 0.5. At layer l+2 target 1
    again: exact on server 1 (1 from server 0, 0 from server 1) or substitute 0
    on server 0 (loss 0.125, free). After the substitute at l+1 the one at l+2
    no longer fits the budget (0.5 + 0.125 > 0.5), so that path costs
    0.125 + 1 against 1 + 0 for the exact one: Phi^(2) = 1. Carrying the loss
    from before the substitute would wrongly let the path cost 0.125."""
    E, M = 2, 2
    t0 = hand_tables(orc, E, M, 0.5, np.zeros((M, M, M), np.float32), pmask=[0b01, 0b10])
    A1 = np.zeros((M, M, M), np.float32); A1[0, 0, 1] = 1.0
    t1 = hand_tables(orc, E, M, 0.5, A1, Q=[[0, 0], [0.25, 0]], Cq=[[0, 0], [0.125, 0]],
                     subst=[0, 0b01], pmask=[0b01, 0b10])
    A2 = np.zeros((M, M, M), np.float32); A2[0, 0, 1] = 1.0; A2[0, 1, 0] = 1.0
    t2 = hand_tables(orc, E, M, 0.5, A2, Q=[[0, 0], [0.125, 0]], subst=[0, 0b01],
                     pmask=[0b01, 0b10])
    P = np.zeros((2, E, E), np.float32)
    P[0, 0, 1] = 1.0                      # l -> l+1: from expert 0 to target 1
    P[1, 0, 1] = P[1, 1, 1] = 1.0         # l+1 -> l+2: to target 1
    assert orc.phi(2, [t0, t1, t2], P, 0, 0, 0, 0.25) == 1.0


def test_phi_continues_from_the_executed_substitute(orc):
    """Eq. 42 two layers ahead: at layer l+1 the next target 1 runs exactly on
    server 1 (cost 1) or as substitute 0 on server 0 (Cq 0.125). The layer
    after follows the transitions of the expert that ran: from 0 to target 0
    (on server 0, cost 0 from server 0), from 1 to target 1 (on server 1, 0
    from server 1, 1 from server 0). So the substitute path costs
    0.125 + 0 and the exact one 1 + 0: Phi^(2) = 0.125. Following the target's
    row instead (1 -> 1) would cost the substitute path 0.125 + 1."""
    E, M = 2, 2
    t0 = hand_tables(orc, E, M, 0.5, np.zeros((M, M, M), np.float32), pmask=[0b01, 0b10])
    A1 = np.zeros((M, M, M), np.float32); A1[0, 0, 1] = 1.0
    t1 = hand_tables(orc, E, M, 0.5, A1, Q=[[0, 0], [0.25, 0]], Cq=[[0, 0], [0.125, 0]],
                     subst=[0, 0b01], pmask=[0b01, 0b10])
    A2 = np.zeros((M, M, M), np.float32); A2[0, 0, 1] = 1.0; A2[0, 1, 0] = 1.0
    t2 = hand_tables(orc, E, M, 0.5, A2, pmask=[0b01, 0b10])
    P = np.zeros((2, E, E), np.float32)
    P[0, 0, 1] = 1.0                      # l -> l+1: from expert 0 to target 1
    P[1, 0, 0] = P[1, 1, 1] = 1.0         # l+1 -> l+2: each expert to itself
    assert orc.phi(2, [t0, t1, t2], P, 0, 0, 0, 0.0) == 0.125


def test_place_load_term_is_weighted_by_lambda1(orc):
    """Eq. 30's score lambda1 b_m / C_m + lambda2 eta_m with lambda1 = 0.25 and
    lambda2 = 0.375. Experts in order 0, 1, 2 (p desc, then importance):
    0 (group 1) -> server 0 (tie at 0, lower server); 1 (group 0) -> server 1
    (0 against 0.25 * 2/4); 2 (group 0): server 0 scores 0.25 * 0.5 = 0.125,
    server 1 (C = 1024, one expert of group 0) 0.25/1024 + 0.375 -> server 0.
    Without the lambda1 weight server 0 would score 0.5 and lose."""
    group = np.array([[1, 0, 0]], np.int32)
    imp = np.array([[3.0, 2.0, 1.0]])
    p = np.array([[2.0, 1.0, 1.0]])
    C = np.array([4.0, 1024.0])
    x, used, rc = orc.place(group, imp, p, C, lambda1=0.25, lambda2=0.375)
    assert rc == 0
    np.testing.assert_array_equal(x[0], [[1, 0, 1], [0, 1, 0]])
    np.testing.assert_array_equal(used, [3.0, 1.0])


def test_place_waiting_list_ties_go_to_the_lower_server(orc):
    """Expert 2 (p = 3) fits no server of capacity 2 and waits; experts 0 and 1
    (p = 2) fill servers 0 and 1. The waiting expert goes to the server with
    the most room; both have 0, so the lower server takes it (and overflows)."""
    group = np.array([[0, 1, 2]], np.int32)
    imp = np.array([[1.0, 1.0, 1.0]])
    p = np.array([[2.0, 2.0, 3.0]])
    C = np.array([2.0, 2.0])
    x, used, rc = orc.place(group, imp, p, C)
    assert rc == orc.CAPACITY
    np.testing.assert_array_equal(x[0], [[1, 0, 1], [0, 1, 0]])
    np.testing.assert_array_equal(used, [5.0, 2.0])


def test_group_hand_example(orc):
    # counts order: 2 (9), 0 (7), 4 (5), 1 (3), 3 (1)
    sim = np.array([[1, .9, .2, .1, .3],
                    [.9, 1, .1, .3, .6],
                    [.2, .1, 1, .8, .1],
                    [.1, .3, .8, 1, .4],
                    [.3, .6, .1, .4, 1]], np.float32)
    cnt = np.array([7, 3, 9, 1, 5], np.int32)
    g, K, dom = orc.group(sim, cnt, 0.5)
    # 2 -> new group 0; 0: sim to 2 is .2 < .5 -> group 1; 4: max(.1, .3) < .5 -> group 2;
    # 1: sims .1 (2), .9 (0), .6 (4) -> joins 0's group 1; 3: .8 (2), .1, .4 -> group 0
    assert K == 3 and list(dom) == [2, 0, 4]
    assert list(g) == [1, 1, 0, 0, 2]
    g2, K2, _ = orc.group(sim, cnt, -1.01)
    assert K2 == 1 and (g2 == 0).all()
    g3, K3, _ = orc.group(sim, cnt, 1.01)
    assert K3 == 5 and sorted(g3) == list(range(5))


def test_group_rule_holds_on_random_inputs(orc):
    rng = np.random.default_rng(20)
    for _ in range(100):
        E = int(rng.integers(2, 12))
        Wt = rng.standard_normal((E, 4))
        sim = (1 - cdist(Wt, Wt, "cosine")).astype(np.float32); np.fill_diagonal(sim, 1)
        cnt = rng.integers(0, 5, E).astype(np.int32)
        th = float(rng.uniform(-0.5, 1.0))
        g, K, dom = orc.group(sim, cnt, th)
        order = sorted(range(E), key=lambda e: (-cnt[e], e))
        made = []
        for j in order:
            if j in dom:
                assert all(sim[j, c] < np.float32(th) for c in made)       # Eq. 24
                assert g[j] == len(made); made.append(j)
            else:
                best = max(sim[j, c] for c in made)
                assert best >= np.float32(th)
                first = next(c for c in made if sim[j, c] == best)          # Eq. 25, tie: earliest
                assert g[j] == made.index(first)


def test_group_clustered_generator_recovers_clusters(orc):
    from paper_2607_17154_gb300 import synth
    E, d, K = 16, 256, 4
    Wr = synth.router_weights(E, d, K, seed=5)
    Xc = synth.calibration(2048, d, seed=5)
    sim = orc.similarity(synth.bits(Wr), synth.bits(Xc))
    cnt = np.ones(E, np.int32)
    for th in (0.3, 0.5, 0.7, 0.9):
        g, KK, _ = orc.group(sim, cnt, th)
        assert KK == K
        cl = synth.cluster_of(E, K)
        for i in range(E):
            for j in range(E):
                assert (g[i] == g[j]) == (cl[i] == cl[j])


def test_importance_closed_forms(orc):
    sim = np.array([[1, .6, 0], [.6, 1, 0], [0, 0, 1]], np.float32)
    group = np.array([0, 0, 1], np.int32)
    cnt = np.array([2, 1, 1], np.int32)
    I = orc.importance(sim, cnt, group, 0.5, 0.5)
    np.testing.assert_allclose(I, [0.5 * 0.5 + 0.5 * 0.8, 0.5 * 0.25 + 0.5 * 0.8, 0.5 * 0.25 + 0.5],
                               rtol=1e-7)
    # unequal weights (Eq. 28: alpha_f on the frequency, alpha_r on the representativeness)
    I2 = orc.importance(sim, cnt, group, 0.75, 0.25)
    np.testing.assert_allclose(I2, [0.75 * 0.5 + 0.25 * 0.8, 0.75 * 0.25 + 0.25 * 0.8,
                                    0.75 * 0.25 + 0.25 * 1.0], rtol=1e-7)
    # no activations at all: the frequency term is 0, the importance alpha_r * rho
    I3 = orc.importance(sim, np.zeros(3, np.int32), group, 0.75, 0.25)
    np.testing.assert_allclose(I3, [0.25 * 0.8, 0.25 * 0.8, 0.25 * 1.0], rtol=1e-7)


def test_place_hand_example_disperses_groups(orc):
    # 4 experts in 2 groups, 2 servers with room for 2 each
    group = np.array([[0, 0, 1, 1]], np.int32)
    I = np.array([[0.9, 0.8, 0.7, 0.6]])
    p = np.ones((1, 4)); C = np.array([2.0, 2.0])
    x, used, rc = orc.place(group, I, p, C)
    assert rc == 0
    # 0 -> server 0 (tie, lower m); 1 -> server 1 (eta); 2 -> server 0 (b/C tie -> eta 0 both, lower);
    # 3 -> server 1 (server 0 full)
    np.testing.assert_array_equal(x[0], [[1, 0, 1, 0], [0, 1, 0, 1]])
    np.testing.assert_array_equal(used, [2, 2])


def test_place_waiting_list_and_capacity(orc):
    group = np.array([[0, 1, 2]], np.int32)
    I = np.array([[0.5, 0.5, 0.5]])
    p = np.array([[2.0, 2.0, 3.0]]); C = np.array([3.0, 4.0])
    x, used, rc = orc.place(group, I, p, C)
    # order by p desc: 2 (3) -> score 0 both -> server 0; 0 (2): feasible {1} -> 1;
    # 1 (2): feasible {1}? b1 = 2, 2+2 <= 4 yes -> 1
    np.testing.assert_array_equal(x[0], [[0, 0, 1], [1, 1, 0]])
    assert rc == 0
    p2 = np.array([[2.0, 2.0, 2.0]]); C2 = np.array([3.0, 3.0])
    x2, used2, rc2 = orc.place(group, I, p2, C2)
    assert x2[0].sum(axis=0).tolist() == [1, 1, 1]          # c.2 still met
    assert rc2 == orc.CAPACITY                               # sum C < sum p
    # unequal room: 2 (p 3) -> server 0, 0 -> server 1, 1 fits nowhere and
    # waits, then goes to the server with the most room left (1: 1.5 > 0)
    x3, used3, rc3 = orc.place(group, I, np.array([[2.0, 2.0, 3.0]]), np.array([3.0, 3.5]))
    np.testing.assert_array_equal(x3[0], [[0, 0, 1], [1, 1, 0]])
    np.testing.assert_array_equal(used3, [3.0, 4.0])
    assert rc3 == orc.CAPACITY


def test_place_invariants_over_layers(orc):
    rng = np.random.default_rng(21)
    for _ in range(50):
        L, E, M = int(rng.integers(1, 5)), int(rng.integers(2, 10)), int(rng.integers(1, 6))
        group = rng.integers(0, 3, (L, E)).astype(np.int32)
        I = rng.random((L, E)); p = rng.integers(1, 4, (L, E)).astype(np.float64)
        C = np.full(M, p.sum() / M * 1.5)
        x, used, rc = orc.place(group, I, p, C)
        assert (x.sum(axis=1) == 1).all()                                   # c.2, one copy
        load = np.einsum("lme,le->m", x.astype(np.float64), p)
        np.testing.assert_allclose(load, used)
        if rc == 0:
            assert (load <= C + 1e-9).all()                                 # c.1
        else:   # only the waiting list may overflow a server
            assert rc == orc.CAPACITY and (load > C).any()


def test_coverage(orc):
    x = np.array([[1, 0, 1, 0], [0, 1, 0, 0]], np.uint8)
    g = np.array([0, 0, 1, 1], np.int32)
    np.testing.assert_array_equal(orc.coverage(x, g, 2), [[1, 1], [1, 0]])


def test_replicate_hand_example(orc):
    # Section IV-C on one layer: groups {0,1} x {2,3}; server 0 covers group 0
    # only, server 1 group 1 only. Benefits (Eq. 33): on server 0, e2 0.15 and
    # e3 0.075; on server 1, e0 0.1 and e1 0.075. One replica each covers the
    # missing group, after which the other candidates' benefit is 0.
    g = np.array([[0, 0, 1, 1]], np.int32)
    I = np.array([[0.4, 0.3, 0.2, 0.1]]); p = np.ones((1, 4))
    x = np.zeros((1, 2, 4), np.uint8); x[0, 0, :2] = 1; x[0, 1, 2:] = 1
    pi = np.array([0.75, 0.25])
    x1, b1, r1 = orc.replicate(g, I, p, np.array([3.0, 3.0]), pi, x, np.array([2.0, 2.0]))
    np.testing.assert_array_equal(x1[0], [[1, 1, 1, 0], [1, 0, 1, 1]])
    np.testing.assert_array_equal(b1, [3, 3]); np.testing.assert_array_equal(r1, [1, 1])
    # Eq. 35: server 1 is full, so only server 0 gets a replica
    x2, b2, r2 = orc.replicate(g, I, p, np.array([3.0, 2.0]), pi, x, np.array([2.0, 2.0]))
    np.testing.assert_array_equal(x2[0], [[1, 1, 1, 0], [0, 0, 1, 1]])
    np.testing.assert_array_equal(r2, [1, 0])
    # a server that no token reaches (pi = 0) has no positive benefit
    x3, _, r3 = orc.replicate(g, I, p, np.array([3.0, 3.0]), np.array([1.0, 0.0]), x,
                              np.array([2.0, 2.0]))
    np.testing.assert_array_equal(r3, [1, 0]); assert x3[0, 1].tolist() == [0, 0, 1, 1]
    # nothing to cover: every server already holds every group
    xf = np.ones((1, 2, 4), np.uint8)
    _, _, r4 = orc.replicate(g, I, p, np.array([9.0, 9.0]), pi, xf, np.array([4.0, 4.0]))
    np.testing.assert_array_equal(r4, [0, 0])


def test_replicate_benefit_is_per_unit_memory_and_ties_go_low(orc):
    # server 0 holds e0 (group 0); group 1 = {e1, e2, e3} with I = .5/.3/.1 and
    # p = 2/1/1: per unit memory e2 (0.3) beats e1 (0.25).
    g = np.array([[0, 1, 1, 1]], np.int32)
    I = np.array([[0.6, 0.5, 0.3, 0.1]]); p = np.array([[1.0, 2.0, 1.0, 1.0]])
    x = np.zeros((1, 1, 4), np.uint8); x[0, 0, 0] = 1
    x1, b1, r1 = orc.replicate(g, I, p, np.array([10.0]), np.array([1.0]), x, np.array([1.0]))
    assert x1[0, 0].tolist() == [1, 0, 1, 0] and b1[0] == 2.0 and r1[0] == 1
    # equal benefits inside a server: the lower expert wins
    I2 = np.array([[0.6, 0.3, 0.3, 0.1]]); p2 = np.ones((1, 4))
    x2, _, _ = orc.replicate(g, I2, p2, np.array([10.0]), np.array([1.0]), x, np.array([1.0]))
    assert x2[0, 0].tolist() == [1, 1, 0, 0]
    # room for one replica, equal benefits in two layers: the lower layer wins
    g3 = np.array([[0, 1], [0, 1]], np.int32)
    I3 = np.array([[0.5, 0.5], [0.5, 0.5]]); p3 = np.ones((2, 2))
    x3 = np.zeros((2, 1, 2), np.uint8); x3[:, 0, 0] = 1
    x4, _, r = orc.replicate(g3, I3, p3, np.array([3.0]), np.array([1.0]), x3, np.array([2.0]))
    assert x4[0, 0].tolist() == [1, 1] and x4[1, 0].tolist() == [1, 0] and r[0] == 1


def per_server_sweep(group, I, p, C, pi, x, used):
    """The greedy of Eqs. 34-35 decomposes over servers (memory and coverage are
    per server, benefits only drop to 0): for each server, visit its
    candidates by benefit desc (ties: layer, expert) and deploy each one whose
    group is still uncovered there and which still fits."""
    L, M, E = x.shape
    x = x.copy(); b = used.astype(np.float64).copy(); reps = np.zeros(M, np.int64)
    for m in range(M):
        cov = {(l, group[l, j]) for l in range(L) for j in range(E) if x[l, m, j]}
        cand = []
        for l in range(L):
            for j in range(E):
                ben = pi[m] * I[l, j] * 1.0 / p[l, j]
                if ben > 0 and (l, group[l, j]) not in cov:
                    cand.append((-ben, l, j))
        for _, l, j in sorted(cand):
            if (l, group[l, j]) in cov or not (b[m] + p[l, j] <= C[m]):
                continue
            x[l, m, j] = 1; b[m] += p[l, j]; cov.add((l, group[l, j])); reps[m] += 1
    return x, b, reps


def test_replicate_invariants_and_per_server_decomposition(orc):
    rng = np.random.default_rng(33)
    for it in range(60):
        L, E, M = int(rng.integers(1, 5)), int(rng.integers(2, 9)), int(rng.integers(1, 6))
        group = rng.integers(0, min(3, E), (L, E)).astype(np.int32)   # group ids < E
        I = rng.random((L, E)) - (0.2 if it % 3 == 0 else 0.0)     # some non-positive
        I[rng.random((L, E)) < 0.2] = 0.5                          # ties
        p = rng.integers(1, 4, (L, E)).astype(np.float64)
        C = np.full(M, p.sum() / M) * rng.uniform(1.0, 3.0, M)
        pi = rng.random(M); pi[rng.random(M) < 0.2] = 0.0
        x0, used0, rc = orc.place(group, np.abs(I), p, C)
        if rc != 0:
            continue
        x, used, reps = orc.replicate(group, I, p, C, pi, x0, used0)
        load = np.einsum("lme,le->m", x.astype(np.float64), p)
        np.testing.assert_allclose(load, used)
        assert (used <= C).all()                                           # Eq. 35
        assert ((x >= x0).all() and int((x - x0).sum()) == int(reps.sum()))
        for l in range(L):
            K = int(group[l].max()) + 1
            c0 = orc.coverage(x0[l], group[l], K); c1 = orc.coverage(x[l], group[l], K)
            new = x[l].astype(int) - x0[l]
            for m in range(M):
                for gg in range(K):
                    nrep = int(new[m][group[l] == gg].sum())
                    assert nrep <= 1 and (nrep == 0 or c0[m, gg] == 0)     # Eq. 32: one per group
                    if c1[m, gg] == 0:                                     # greedy stopped for a reason
                        for j in np.nonzero(group[l] == gg)[0]:
                            assert pi[m] * I[l, j] <= 0 or used[m] + p[l, j] > C[m]
        xs, bs, rs = per_server_sweep(group, I, p, C, pi, x0, used0)
        np.testing.assert_array_equal(x, xs)
        np.testing.assert_array_equal(used, bs)
        np.testing.assert_array_equal(reps, rs)


def test_replicate_with_ample_memory_covers_every_group_everywhere(orc):
    rng = np.random.default_rng(4)
    L, E, M = 3, 8, 4
    group = rng.integers(0, 4, (L, E)).astype(np.int32)
    I = rng.random((L, E)) + 0.1; p = np.ones((L, E))
    x0, used0, rc = orc.place(group, I, p, np.full(M, L * E / M))
    assert rc == 0
    x, used, reps = orc.replicate(group, I, p, np.full(M, 1e9), np.full(M, 0.25), x0, used0)
    uncovered = 0
    for l in range(L):
        K = int(group[l].max()) + 1
        present = np.unique(group[l])
        c0 = orc.coverage(x0[l], group[l], K); c1 = orc.coverage(x[l], group[l], K)
        assert (c1[:, present] == 1).all()
        uncovered += int((c0[:, present] == 0).sum())
    assert int(reps.sum()) == uncovered


def _sim_params():
    # dyadic values, so every delay below is exact in fp64; B and tau asymmetric
    F = np.array([4.0, 2.0, 8.0])
    B = np.array([[1.0, 2.0, 8.0], [4.0, 1.0, 1.0], [16.0, 2.0, 1.0]])
    tau = np.array([[0.0, 0.5, 0.25], [0.25, 0.0, 2.0], [0.125, 1.0, 0.0]])
    return F, B, tau


def test_trajectory_cost_hand_example(orc):
    # Eqs. 13-20 on two layers. Token 0 (home 0): layer 1 slot 0 on server 1
    # (transfer 8/2 + 0.5, compute 1/2), slot 1 substitutes expert 3 for 2 on
    # server 0 (compute 1/4); the token is then on server 1 (slot 0). Layer 2:
    # slot 0 on server 1 (compute 1/2), slot 1 on server 2 (transfer 8/1 + 2,
    # compute 1/8). Token 1 (home 2) stays on server 2 with exact experts.
    F, B, tau = _sim_params()
    E, L, T, k = 4, 2, 2, 2
    target = np.array([[[1, 2], [0, 1]], [[0, 3], [2, 3]]], np.int32)
    chosen = np.array([[[1, 3], [0, 1]], [[0, 3], [2, 3]]], np.int32)
    server = np.array([[[1, 0], [2, 2]], [[1, 2], [2, 2]]], np.uint8)
    home = np.array([0, 2], np.uint8)
    Qtab = np.zeros((L, E, E), np.float32); Qtab[0, 2, 3] = 0.125; Qtab[1, 0, 3] = 0.5
    d, q, n = orc.trajectory_cost(target, chosen, server, home, F, B, tau, 8.0, 1.0, Qtab)
    assert d[0] == (4.5 + 0.5 + 0.25) + (0.5 + 10.0 + 0.125)
    assert d[1] == 4 * 0.125
    assert q.tolist() == [0.125, 0.0] and n.tolist() == [2, 0]


def test_trajectory_cost_agrees_with_the_selection_cost_table(orc):
    # Eq. 37's delay term, built by orc_tables from the same server parameters,
    # equals omega_T * (Eqs. 13-15 delay) / d_ref(a) for each slot of a
    # one-layer trajectory that starts at home (up to the tables' fp32 rounding).
    rng = np.random.default_rng(7)
    E, M, k, T = 8, 4, 2, 200
    F = rng.uniform(20e12, 110e12, M)
    B = rng.uniform(1e8, 1.25e9, (M, M)); tau = rng.uniform(2e-4, 2e-2, (M, M))
    np.fill_diagonal(tau, 0.0)
    z, c, wT = 8192.0, 3.5e8, 0.5
    sim = np.eye(E, dtype=np.float32); group = np.arange(E, dtype=np.int32)
    x = (rng.random((M, E)) < 0.5).astype(np.uint8); x[0] = 1
    tab = orc.tables(sim, group, x, 0.5, 0.1, F, B, tau, z, c, wT, 0.5)
    idx, _ = orc.topk(rng.standard_normal((T, E)).astype(np.float32), k)
    home = rng.integers(0, M, T).astype(np.uint8)
    ch, sv, _, _, _ = orc.select(idx, tab, home, home.copy(), np.zeros(T, np.float32))
    d, q, n = orc.trajectory_cost(idx[None], ch[None], sv[None], home, F, B, tau, z, c,
                                  tab.Qtab[None])
    A = tab.A.reshape(M, M, M)
    for t in range(T):
        a = home[t]
        want = sum(float(A[a, a, m]) for m in sv[t])
        np.testing.assert_allclose(wT * d[t] / (c / F[a]), want, rtol=1e-6)
        assert n[t] == int((sv[t] != a).sum()) and q[t] == 0.0


def test_utility_and_weight_adaptation_closed_forms(orc):
    T = 8
    d = np.full(T, 3.0); q = np.full(T, 0.25)
    # delay equal to the exact-execution reference, half the budget used
    U, tb, qb, wT, wQ = orc.utility(d, d, q, 0.5, 0.75, 0.25, 0.125)
    assert (tb, qb) == (1.0, 0.5)
    assert U == 0.75 * 8 + 0.25 * 4
    assert wQ == 0.25 + 0.125 * (0.5 - 1.0) and wT == 1.0 - wQ
    # the projection onto [0, 1]
    assert orc.utility(d, d, q, 0.5, 0.5, 0.5, 4.0)[4] == 0.0
    assert orc.utility(d, 2 * d, 4 * q, 0.5, 0.5, 0.5, 4.0)[4] == 1.0
    # random values against an exactly rounded sum
    import math
    rng = np.random.default_rng(3)
    d = rng.uniform(1, 3, 500); r = rng.uniform(1, 2, 500); q = rng.uniform(0, 0.1, 500)
    U, tb, qb, wT, wQ = orc.utility(d, r, q, 0.1, 0.6, 0.4, 0.05)
    st = math.fsum(d / r); sq = math.fsum(q / 0.1)
    np.testing.assert_allclose([U, tb, qb], [0.6 * st + 0.4 * sq, st / 500, sq / 500], rtol=1e-12)
    np.testing.assert_allclose(wQ, 0.4 + 0.05 * (sq / 500 - st / 500), rtol=1e-12)


def test_group_threshold_is_strict_and_ties_go_to_the_earlier_dominant(orc):
    cnt = np.array([3, 2, 1], np.int32)            # visiting order 0, 1, 2
    # Sim(1, 0) == theta: Eq. 24 needs max Sim < theta for a new dominant, so 1 joins 0
    sim = np.array([[1, .5, .3], [.5, 1, .3], [.3, .3, 1]], np.float32)
    g, K, dom = orc.group(sim, cnt, 0.5)
    assert K == 2 and list(g) == [0, 0, 1]
    # 0 and 1 are dominants (Sim .1 < .3); 2 is equally similar to both (.6):
    # Eq. 25's argmax tie goes to the earlier dominant
    sim2 = np.array([[1, .1, .6], [.1, 1, .6], [.6, .6, 1]], np.float32)
    g2, K2, dom2 = orc.group(sim2, cnt, 0.3)
    assert K2 == 2 and list(dom2) == [0, 1] and g2[2] == 0
    # zeros of either sign are equal similarities: 2 is -0 to dominant 0 and +0
    # to dominant 1 (0 and 1 at -0.5 from each other, threshold -0.25), so the
    # tie goes to the earlier dominant; with the signs swapped it is the same
    for z0, z1 in ((-0.0, 0.0), (0.0, -0.0)):
        sim3 = np.array([[1, -.5, z0], [-.5, 1, z1], [z0, z1, 1]], np.float32)
        g3, K3, dom3 = orc.group(sim3, cnt, -0.25)
        assert K3 == 2 and list(dom3) == [0, 1] and g3[2] == 0, (z0, z1, g3)


def test_place_disperses_same_group_experts_even_when_load_alone_would_not(orc):
    # importance order 0 (g0), 2 (g1), 1 (g0), 3 (g1) on 2 servers of capacity 4:
    # load balance alone would put 0 and 1 together; the eta term of Eq. 30
    # sends each server one expert of each group
    group = np.array([[0, 0, 1, 1]], np.int32)
    I = np.array([[0.9, 0.7, 0.8, 0.6]])
    x, used, rc = orc.place(group, I, np.ones((1, 4)), np.array([4.0, 4.0]))
    assert rc == 0
    np.testing.assert_array_equal(x[0], [[1, 0, 0, 1], [0, 1, 1, 0]])


# --------------------------------------------------------------------------
# Look-ahead selection (Eqs. 41-43)

def test_transitions_brute_force(orc):
    rng = np.random.default_rng(30)
    N, L, E, kf = 40, 4, 6, 2
    logits = rng.standard_normal((N, L, E)).astype(np.float32)
    logits[0, 1, :] = 0.5                       # ties
    logits[:, 0, 5] = -10.0                     # expert 5 never in the top-2 at layer 0
    cnt, P = orc.transitions(logits, kf)
    ref = np.zeros((L - 1, E, E), np.int64)
    for n in range(N):
        for l in range(L - 1):
            for a in brute_topk(list(logits[n, l]), kf):
                for b in brute_topk(list(logits[n, l + 1]), kf):
                    ref[l, a, b] += 1
    np.testing.assert_array_equal(cnt, ref)
    rows = ref.sum(axis=2, keepdims=True)
    np.testing.assert_allclose(P, np.where(rows > 0, ref / np.maximum(rows, 1), 0), rtol=1e-7)
    assert cnt.sum() == (L - 1) * N * kf * kf
    # a row without transitions is 0 (Eq. 41's quotient has no denominator there)
    assert (cnt[0, 5] == 0).all() and (P[0, 5] == 0).all()


def _rand_tables(orc, rng, E, M, kgroups, tau_scale=1.0):
    Wt = rng.standard_normal((E, 5)); Wt[:, 0] += 3.0 * (np.arange(E) % kgroups)
    sim = (1 - cdist(Wt, Wt, "cosine")).astype(np.float32); np.fill_diagonal(sim, 1.0)
    group = (np.arange(E) % kgroups).astype(np.int32)
    x = (rng.random((M, E)) < 0.4).astype(np.uint8)
    for e in range(E):
        if not x[:, e].any():
            x[rng.integers(M), e] = 1
    F, B, tau = _params(rng, M)
    return orc.tables(sim, group, x, float(rng.choice([0.0, 0.4])), float(rng.choice([0.1, 0.3])),
                      F, B, tau * tau_scale, 2048.0, 1e9, 0.5, 0.5), sim


def test_lookahead_horizon_one_is_the_myopic_selection(orc):
    rng = np.random.default_rng(31)
    for _ in range(40):
        E, M, k, T = int(rng.integers(2, 7)), int(rng.integers(1, 4)), 1, 12
        k = int(rng.integers(1, min(E, 3) + 1))
        tab, _ = _rand_tables(orc, rng, E, M, 2, tau_scale=float(rng.choice([1e-4, 1.0])))
        idx = np.array([rng.permutation(E)[:k] for _ in range(T)], np.int32)
        home = rng.integers(0, M, T).astype(np.uint8)
        loc = rng.integers(0, M, T).astype(np.uint8)
        qhat = (rng.random(T) * 0.05).astype(np.float32)
        a = orc.select(idx, tab, home, loc, qhat)
        b = orc.select_lookahead(idx, [tab], None, home, loc, qhat)
        for u, v in zip(a, b):
            np.testing.assert_array_equal(u, v)


def brute_lookahead_h2(idx, t0, t1, P1, home, loc, qhat):
    """Eq. 43 with H = 2, Eq. 42 enumerated over every (target k', server m',
    executed expert k'') triple of the next layer; fp32 as the paper's
    reading fixes it (each product and sum rounded once)."""
    f32 = np.float32
    T, k = idx.shape
    E, M = t0.E, t0.M
    out = [np.zeros((T, k), np.int32), np.zeros((T, k), np.uint8), np.zeros((T, k), np.uint8)]
    loc2 = loc.copy(); q2 = qhat.copy()

    def feasible(t, target, qacc, taken):
        for m in range(M):
            for kk in range(E):
                if not (int(t.pmask[kk]) >> m) & 1:
                    continue
                if kk != target:
                    if not (int(t.subst[target]) >> kk) & 1 or kk in taken:
                        continue
                    if not f32(qacc + t.Qtab[target, kk]) <= t.qbar:
                        continue
                yield m, kk

    for ti in range(T):
        a, s, q = int(home[ti]), int(loc[ti]), f32(qhat[ti])
        taken = set(int(v) for v in idx[ti])
        for j in range(k):
            r = int(idx[ti, j])
            cands = []
            for m, kk in feasible(t0, r, q, taken):
                g = f32(t0.A[a, s, m] + (f32(0) if kk == r else t0.Cq[r, kk]))
                qn = q if kk == r else f32(q + t0.Qtab[r, kk])
                phi = f32(0)
                for kt in range(E):
                    p = P1[kk, kt]
                    if p == 0:
                        continue
                    best = min(f32(t1.A[a, m, m2] + (f32(0) if k2 == kt else t1.Cq[kt, k2]))
                               for m2, k2 in feasible(t1, kt, qn, set()))
                    phi = f32(phi + f32(p * best))
                cands.append((f32(g + phi), kk != r, m != s, m, kk))
            _, sub, away, m, kk = min(cands)
            out[0][ti, j] = kk; out[1][ti, j] = m; out[2][ti, j] = 2 * away + sub
            if sub:
                taken.add(kk); q = f32(q + t0.Qtab[r, kk])
            if j == 0:
                loc2[ti] = m
        q2[ti] = q
    return out[0], out[1], out[2], loc2, q2


def test_lookahead_h2_matches_brute_force(orc):
    rng = np.random.default_rng(32)
    changed = 0
    for trial in range(60):
        E, M = int(rng.integers(2, 6)), int(rng.integers(1, 4))
        k = int(rng.integers(1, min(E, 2) + 1)); T = 8
        scale = float(rng.choice([1e-4, 1e-2, 1.0]))
        t0, _ = _rand_tables(orc, rng, E, M, 2, tau_scale=scale)
        t1, _ = _rand_tables(orc, rng, E, M, 2, tau_scale=scale)
        t1.qbar = t0.qbar
        P1 = rng.random((E, E)).astype(np.float32)
        P1[P1 < 0.3] = 0
        P1 = (P1 / np.maximum(P1.sum(axis=1, keepdims=True), 1e-9)).astype(np.float32)
        idx = np.array([rng.permutation(E)[:k] for _ in range(T)], np.int32)
        home = rng.integers(0, M, T).astype(np.uint8)
        loc = rng.integers(0, M, T).astype(np.uint8)
        qhat = (rng.random(T) * 0.05).astype(np.float32)
        got = orc.select_lookahead(idx, [t0, t1], P1[None], home, loc, qhat)
        ref = brute_lookahead_h2(idx, t0, t1, P1, home, loc, qhat)
        for u, v in zip(got, ref):
            np.testing.assert_array_equal(u, v)
        myo = orc.select(idx, t0, home, loc, qhat)
        changed += int((myo[0] != got[0]).sum() + (myo[1] != got[1]).sum())
    assert changed > 0   # the look-ahead did change some decisions


def _feasible(t, target, qacc, taken):
    """Eq. 40 from its definition: (server, executed expert) pairs where the
    expert is placed, is the target or an unused within-budget substitute."""
    f32 = np.float32
    for m in range(t.M):
        for kk in range(t.E):
            if not (int(t.pmask[kk]) >> m) & 1:
                continue
            if kk != target:
                if not (int(t.subst[target]) >> kk) & 1 or kk in taken:
                    continue
                if not f32(qacc + t.Qtab[target, kk]) <= t.qbar:
                    continue
            yield m, kk


def brute_phi(h, tabs, Ps, a, m, kx, qacc):
    """Eq. 42's Phi^(h) by recursive enumeration (tabs[len - h] is the next
    layer, Ps[len - 1 - h] the transition into it), fp32."""
    f32 = np.float32
    if h == 0:
        return f32(0)
    t1, P = tabs[len(tabs) - h], Ps[len(tabs) - 1 - h]
    acc = f32(0)
    for kt in range(t1.E):
        p = P[kx, kt]
        if p == 0:
            continue
        best = f32(np.inf)
        for m2, k2 in _feasible(t1, kt, qacc, set()):
            c = f32(t1.A[a, m, m2] + (f32(0) if k2 == kt else t1.Cq[kt, k2]))
            if h > 1:
                qn = qacc if k2 == kt else f32(qacc + t1.Qtab[kt, k2])
                c = f32(c + brute_phi(h - 1, tabs, Ps, a, m2, k2, qn))
            best = min(best, c)
        acc = f32(acc + f32(p * best))
    return acc


def brute_lookahead(idx, tabs, Ps, home, loc, qhat):
    """Eq. 43 with any horizon H = len(tabs): Eq. 42's cost-to-go enumerated
    recursively over every (target k', server m', executed expert k'') path of
    the future layers, straight from the feasibility rule of Eq. 40 (no
    substitute bitmask or placement-mask shortcut), fp32 as the reading fixes it."""
    f32 = np.float32
    T, k = idx.shape
    t0 = tabs[0]
    E, M = t0.E, t0.M
    out = [np.zeros((T, k), np.int32), np.zeros((T, k), np.uint8), np.zeros((T, k), np.uint8)]
    loc2 = loc.copy(); q2 = qhat.copy()

    def feasible(t, target, qacc, taken):
        for m in range(M):
            for kk in range(E):
                if not (int(t.pmask[kk]) >> m) & 1:
                    continue
                if kk != target:
                    if not (int(t.subst[target]) >> kk) & 1 or kk in taken:
                        continue
                    if not f32(qacc + t.Qtab[target, kk]) <= t.qbar:
                        continue
                yield m, kk

    def phi(h, a, m, kx, qacc):
        return brute_phi(h, tabs, Ps, a, m, kx, qacc)

    H = len(tabs)
    for ti in range(T):
        a, s, q = int(home[ti]), int(loc[ti]), f32(qhat[ti])
        taken = set(int(v) for v in idx[ti])
        for j in range(k):
            r = int(idx[ti, j])
            cands = []
            for m, kk in feasible(t0, r, q, taken):
                g = f32(t0.A[a, s, m] + (f32(0) if kk == r else t0.Cq[r, kk]))
                qn = q if kk == r else f32(q + t0.Qtab[r, kk])
                cost = f32(g + phi(H - 1, a, m, kk, qn)) if H > 1 else g
                cands.append((cost, kk != r, m != s, m, kk))
            _, sub, away, m, kk = min(cands)
            out[0][ti, j] = kk; out[1][ti, j] = m; out[2][ti, j] = 2 * away + sub
            if sub:
                taken.add(kk); q = f32(q + t0.Qtab[r, kk])
            if j == 0:
                loc2[ti] = m
        q2[ti] = q
    return out[0], out[1], out[2], loc2, q2


@pytest.mark.parametrize("H,trials", [(3, 30), (4, 8)])
def test_lookahead_deep_horizons_match_brute_force(orc, H, trials):
    """The paper's default horizon H = 3 (and H = 4) against the recursive
    enumeration, with budgets tight enough that future substitutes become
    infeasible along some paths."""
    rng = np.random.default_rng(40 + H)
    for trial in range(trials):
        E, M = int(rng.integers(2, 5)), int(rng.integers(1, 4))
        k = int(rng.integers(1, min(E, 2) + 1)); T = 6
        scale = float(rng.choice([1e-4, 1e-2, 1.0]))
        tabs = [_rand_tables(orc, rng, E, M, 2, tau_scale=scale)[0] for _ in range(H)]
        for t in tabs[1:]:
            t.qbar = tabs[0].qbar
        Ps = []
        for _ in range(H - 1):
            P = rng.random((E, E)).astype(np.float32)
            P[P < 0.3] = 0
            Ps.append((P / np.maximum(P.sum(axis=1, keepdims=True), 1e-9)).astype(np.float32))
        idx = np.array([rng.permutation(E)[:k] for _ in range(T)], np.int32)
        home = rng.integers(0, M, T).astype(np.uint8)
        loc = rng.integers(0, M, T).astype(np.uint8)
        qhat = (rng.random(T) * float(rng.choice([0.05, 0.25]))).astype(np.float32)
        got = orc.select_lookahead(idx, tabs, np.stack(Ps), home, loc, qhat)
        ref = brute_lookahead(idx, tabs, Ps, home, loc, qhat)
        for u, v in zip(got, ref):
            np.testing.assert_array_equal(u, v)


def test_cost_to_go_values_match_brute_force(orc):
    """Phi^(h), h = 1..3, value for value (the same fp32 operations), so that a
    deeper level reading the wrong layer or transition matrix shows even where
    it would not change a decision."""
    rng = np.random.default_rng(47)
    n = 0
    for trial in range(12):
        E, M = int(rng.integers(2, 5)), int(rng.integers(1, 4))
        H = 4
        scale = float(rng.choice([1e-3, 1.0]))
        tabs = [_rand_tables(orc, rng, E, M, 2, tau_scale=scale)[0] for _ in range(H)]
        for t in tabs[1:]:
            t.qbar = tabs[0].qbar
        Ps = []
        for _ in range(H - 1):
            P = rng.random((E, E)).astype(np.float32)
            P[P < 0.3] = 0
            Ps.append((P / np.maximum(P.sum(axis=1, keepdims=True), 1e-9)).astype(np.float32))
        for h in (1, 2, 3):
            for _ in range(6):
                a, m, kx = int(rng.integers(M)), int(rng.integers(M)), int(rng.integers(E))
                q = float(np.float32(rng.random() * 0.2))
                want = brute_phi(h, tabs[:h + 1], Ps[:h], a, m, kx, np.float32(q))
                got = orc.phi(h, tabs[:h + 1], np.stack(Ps[:h]), a, m, kx, q)
                assert np.float32(got) == want or (np.isinf(got) and np.isinf(want)), (h, got, want)
                n += 1
    assert n == 12 * 3 * 6


def test_lookahead_moves_the_token_where_the_next_layer_is_cheap(orc):
    """Hand case (Eqs. 37-43): the target r is only on server 1; its substitute
    s2 is local on server 0. Myopically the local substitute is cheaper
    (1 + 0.5 < 5), but every next-layer target lives on server 1 only, so with
    H = 2 moving now costs 5 + 1 < 1.5 + 5 and the token goes to server 1."""
    E, M = 3, 2
    A = np.array([[[1, 5], [5, 1]], [[1, 5], [5, 1]]], np.float32)
    Q = np.array([[0, .2, .2], [.2, 0, .2], [.2, .2, 0]], np.float32)
    Cq = np.where(Q > 0, 0.5, 0).astype(np.float32)
    t0 = orc.Tables(Q, Cq, np.array([0b010, 0b001, 0], np.uint64), A,
                    np.array([0b10, 0b01, 0b10], np.uint32), 1.0, E, M)
    t1 = orc.Tables(Q, Cq, np.zeros(E, np.uint64), A, np.array([0b10, 0b10, 0b10], np.uint32), 1.0,
                    E, M)
    P = np.zeros((1, E, E), np.float32); P[0, :, 2] = 1.0
    idx = np.array([[0]], np.int32)
    home = np.array([0], np.uint8)
    myo = orc.select(idx, t0, home, home.copy(), np.zeros(1, np.float32))
    assert myo[0][0, 0] == 1 and myo[1][0, 0] == 0          # local substitute
    la = orc.select_lookahead(idx, [t0, t1], P, home, home.copy(), np.zeros(1, np.float32))
    assert la[0][0, 0] == 0 and la[1][0, 0] == 1            # remote exact
    assert la[3][0] == 1                                     # the token moved (Eq. 44)


def test_group_and_place_with_nan_similarities(orc):
    """NaN similarities (bad inputs) follow the scan's own rule: an expert joins
    the first dominant when its similarity to it is NaN (NaN < theta is
    false, and nothing strictly exceeds NaN), and otherwise a NaN never wins.
    The importance of such experts is NaN; the placement order puts NaN after
    every number (a total order), so the placement stays a permutation."""
    # counts order: 0, 1, 2, 3; dominant 0 first
    sim = np.array([[1, .9, .2, np.nan],
                    [.9, 1, .1, .3],
                    [.2, .1, 1, .8],
                    [np.nan, .3, .8, 1]], np.float32)
    cnt = np.array([9, 7, 5, 3], np.int32)
    g, K, dom = orc.group(sim, cnt, 0.5)
    # 0 -> group 0; 1 joins 0 (.9); 2: .2 < .5 -> group 1 (dominant 2);
    # 3: NaN to dominant 0 first -> joins group 0 although .8 to dominant 2 is larger
    assert K == 2 and list(dom[:2]) == [0, 2] and list(g) == [0, 0, 1, 0]
    sim2 = sim.copy(); sim2[3, 0] = sim2[0, 3] = 0.1; sim2[3, 2] = sim2[2, 3] = np.nan
    g2, K2, _ = orc.group(sim2, cnt, 0.5)
    # 3: .1 to dominant 0, NaN to dominant 2 (never wins) -> best .1 < .5 -> new group 2
    assert K2 == 3 and list(g2) == [0, 0, 1, 2]
    imp = orc.importance(sim, cnt, g)
    # rho of 0 and 3 averages the NaN pair Sim(0,3); expert 1's group mean does not include it
    assert np.isnan(imp[[0, 3]]).all() and np.isfinite(imp[[1, 2]]).all()
    assert imp[2] == pytest.approx(0.5 * 5 / 24 + 0.5) and imp[1] == pytest.approx(0.5 * 7 / 24 + 0.5 * 2.2 / 3)
    # placement order: 2 (I .604), 1 (.5125), then the NaN importances 0, 3 by index.
    # 2 -> server 0 (both empty, ties to the lower m); 1 -> server 1 (0.25 against 0);
    # 0 (group 0) -> server 0 (0.25 + 0 against 0.25 + 0.5 for expert 1's group on 1);
    # 3 -> server 1 (server 0 is full)
    L, E, M = 1, 4, 2
    x, used, rc = orc.place(g[None], imp[None], np.ones((1, E)), np.full(M, 2.0))
    assert rc == 0 and list(used) == [2.0, 2.0]
    assert x[0].tolist() == [[1, 0, 1, 0], [0, 1, 0, 1]]
    x2, _, _ = orc.place(g[None], imp[None], np.ones((1, E)), np.full(M, 2.0))
    assert (x2 == x).all()                                          # deterministic
