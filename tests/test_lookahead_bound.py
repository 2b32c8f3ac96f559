"""The budget bound that lets the look-ahead kernels read the deepest cost-to-go
from a per-token table (Eq. 42), checked on the oracle's Phi.

Phi^(h)(m, k, q) depends on the accumulated loss q only through its budget
checks fl(q + Q) <= Qbar (Eq. 44). Let Qmax(k) be the largest substitute loss
that Phi^(1)(., k) can consider (targets k' with P(k -> k') != 0, -inf when
there is none). Since fp32 addition rounds monotonically and q >= 0,
fl(q + Qmax(k)) <= Qbar means every check passes at q as at 0, so
Phi^(1)(m, k, q) == Phi^(1)(m, k, 0) bit for bit; one level up, Phi^(2) needs
the bound of its own level and, for the loss entering the level below, that
level's largest loss too. These tests draw random tables and losses, confirm
the equality wherever the bound holds, and confirm that the values do differ
for some losses that break it (the bound is not vacuous)."""
import numpy as np
import pytest

import oracle
from paper_2607_17154_gb300 import synth


def f32add(a, b):
    return np.float32(np.float32(a) + np.float32(b))


def random_tables(rng, n, E, M, qbar):
    tabs = []
    for l in range(n):
        Wt = rng.standard_normal((E, 5))
        Wt[:, 0] += 2.0 * (np.arange(E) % 3)
        Wn = Wt / np.linalg.norm(Wt, axis=1, keepdims=True)
        sim = (Wn @ Wn.T).astype(np.float32)
        np.fill_diagonal(sim, 1.0)
        group = (np.arange(E) % 3).astype(np.int32)
        x = (rng.random((M, E)) < 0.4).astype(np.uint8)
        for e in range(E):
            if not x[:, e].any():
                x[rng.integers(M), e] = 1
        sp = synth.server_params(M, 1024, 2048, seed=int(rng.integers(1 << 30)))
        tabs.append(oracle.tables(sim, group, x, 0.1, qbar, sp.F, sp.B, sp.tau, sp.z, sp.c,
                                  sp.omega_T, sp.omega_Q))
    return tabs


def random_P(rng, n, E):
    P = rng.random((n, E, E)).astype(np.float32)
    P[P < 0.4] = 0
    return (P / np.maximum(P.sum(axis=2, keepdims=True), 1e-9)).astype(np.float32)


def qmax_of(tab, P, kx):
    """The largest substitute loss Phi^(1) from expert kx on tables tab and
    transitions P can consider (-inf: none)."""
    E = tab.E
    mx = np.float32(-np.inf)
    for kt in range(E):
        if P[kx, kt] == 0:
            continue
        for k3 in range(E):
            if (int(tab.subst[kt]) >> k3) & 1:
                mx = max(mx, tab.Qtab[kt, k3])
    return np.float32(mx)


def losses(rng, qbar, n):
    """Accumulated losses in [0, qbar], with exact 0 and qbar among them."""
    q = list((rng.random(n - 2) * qbar).astype(np.float32))
    return [np.float32(0.0), np.float32(qbar)] + q


@pytest.mark.parametrize("seed", range(4))
def test_phi1_is_its_zero_loss_value_when_the_bound_holds(seed):
    rng = np.random.default_rng(100 + seed)
    E, M = 8, 4
    qbar = np.float32(0.6)
    t = random_tables(rng, 2, E, M, qbar)      # layers l+1 (not read by Phi^(1)) and l+2
    P = random_P(rng, 1, E)                     # P_{l+1}
    held = differ = 0
    for a in range(M):
        for m2 in range(M):
            for k2 in range(E):
                qm = qmax_of(t[1], P[0], k2)
                z = oracle.phi(1, t, P, a, m2, k2, 0.0)
                for q2 in losses(rng, qbar, 6):
                    v = oracle.phi(1, t, P, a, m2, k2, float(q2))
                    if f32add(q2, qm) <= qbar:
                        held += 1
                        assert np.float32(v).tobytes() == np.float32(z).tobytes(), (a, m2, k2, q2)
                    elif v != z:
                        differ += 1
    assert held > 100 and differ > 0, (held, differ)


@pytest.mark.parametrize("seed", range(3))
def test_phi2_is_its_zero_loss_value_when_both_bounds_hold(seed):
    rng = np.random.default_rng(200 + seed)
    E, M = 6, 3
    qbar = np.float32(0.8)
    t = random_tables(rng, 3, E, M, qbar)      # layers l+1 (not read), l+2, l+3
    P = random_P(rng, 2, E)                     # P_{l+1}, P_{l+2}
    qmaxL1 = max(qmax_of(t[2], P[1], k3) for k3 in range(E))
    held = differ = 0
    for a in range(M):
        for m2 in range(M):
            for k2 in range(E):
                qm2 = qmax_of(t[1], P[0], k2)
                z = oracle.phi(2, t, P, a, m2, k2, 0.0)
                for q2 in losses(rng, qbar, 6):
                    qa = f32add(q2, qm2)
                    q3max = q2 if qm2 == -np.inf else qa   # largest loss entering level 1
                    v = oracle.phi(2, t, P, a, m2, k2, float(q2))
                    if qa <= qbar and f32add(q3max, qmaxL1) <= qbar:
                        held += 1
                        assert np.float32(v).tobytes() == np.float32(z).tobytes(), (a, m2, k2, q2)
                    elif v != z:
                        differ += 1
    assert held > 20 and differ > 0, (held, differ)
