"""GPU parity of the offline plan (similarity, counts, grouping, placement;
Eqs. 3-6, 24-31) and of the whole-layer entry point, against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_17154_gb300 import binding as B
from paper_2607_17154_gb300 import synth
from paper_2607_17154_gb300.layer import build_tables
from tests.helpers import assert_close_bf16
from tests.test_gpu_path import random_tables_case

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.lib()
    yield
    code, detail = B.ordermoe_device_error()
    assert code == 0, "device error word %d (detail %d) after tests" % (code, detail)


def gpu_similarity(Wr_stack, Xcal, kf):
    L, E, d = Wr_stack.shape
    N = Xcal.shape[0]
    sim = torch.empty(L, E, E, dtype=torch.float32, device=DEV)
    counts = torch.empty(L, E, dtype=torch.int32, device=DEV)
    ws = torch.empty(B.ordermoe_similarity_workspace_bytes(L, E, N), dtype=torch.uint8, device=DEV)
    B.ordermoe_similarity(Wr_stack.to(DEV).contiguous(), Xcal.to(DEV), L, E, d, N, kf, sim, counts, ws)
    torch.cuda.synchronize()
    return sim.cpu().numpy(), counts.cpu().numpy()


@pytest.mark.parametrize("L,E,d,N,kf,K", [(1, 8, 256, 4096, 2, 2), (3, 64, 512, 3000, 6, 8),
                                          (2, 16, 128, 700, 3, 4), (5, 32, 256, 1029, 4, 4),
                                          (2, 12, 128, 1000, 3, 3), (3, 48, 256, 2100, 6, 6)])
def test_similarity_matches_oracle(L, E, d, N, kf, K):
    Wr = torch.stack([synth.router_weights(E, d, K, seed=10 + l) for l in range(L)])
    Xcal = synth.calibration(N, d, seed=L * 100 + E)
    sim, counts = gpu_similarity(Wr, Xcal, kf)
    for l in range(L):
        ref, H = oracle.similarity(synth.bits(Wr[l]), synth.bits(Xcal), return_H=True)
        np.testing.assert_allclose(sim[l], ref, atol=2e-5, rtol=0)
        assert (np.diag(sim[l]) == 1).all()
        ref_counts = oracle.expert_counts(np.ascontiguousarray(H.T), kf)
        assert counts[l].sum() == N * kf
        # counts from fp32 logits of different summation order: equal up to near ties
        assert np.abs(counts[l] - ref_counts).sum() <= max(2, N // 500), (counts[l], ref_counts)


@pytest.mark.parametrize("L,E,d,N,kf", [(3, 64, 512, 3000, 6), (2, 16, 128, 700, 3), (2, 12, 128, 1000, 3)])
def test_similarity_no_logits_same_results(L, E, d, N, kf):
    # the entry point that skips the fp32 logits gives the same sim and counts bit for bit
    Wr = torch.stack([synth.router_weights(E, d, 4, seed=20 + l) for l in range(L)]).to(DEV).contiguous()
    Xcal = synth.calibration(N, d, seed=7 * L + E).to(DEV)
    ws = torch.empty(B.ordermoe_similarity_workspace_bytes(L, E, N), dtype=torch.uint8, device=DEV)
    sim_a = torch.empty(L, E, E, dtype=torch.float32, device=DEV)
    cnt_a = torch.empty(L, E, dtype=torch.int32, device=DEV)
    B.ordermoe_similarity(Wr, Xcal, L, E, d, N, kf, sim_a, cnt_a, ws)
    logits = ws[: N * L * E * 4].view(torch.float32).view(N, L * E).clone()
    ws.fill_(0xFF)  # the logits region is not rewritten by the second call
    sim_b = torch.empty_like(sim_a)
    cnt_b = torch.empty_like(cnt_a)
    B.ordermoe_similarity_no_logits(Wr, Xcal, L, E, d, N, kf, sim_b, cnt_b, ws)
    torch.cuda.synchronize()
    assert torch.equal(sim_a, sim_b) and torch.equal(cnt_a, cnt_b)
    assert torch.isfinite(logits).all()
    region = ws[: N * L * E * 4]
    if E in (8, 16, 32, 64):  # tensor-core path: the logits are skipped
        assert (region == 0xFF).all()
    else:  # the CUDA-core path needs them and keeps them
        assert torch.equal(region.view(torch.float32).view(N, L * E), logits)


@pytest.mark.parametrize("kf", [1, 6, 8, 9])
def test_similarity_counts_exact_with_tied_logits(kf):
    """The counts of Eq. 5 equal the oracle's on the kernel's own fp32 logits,
    bit for bit, with exact ties: duplicated router rows give equal logits for
    every token, so equal logits straddle the top-k boundary (the lower index
    wins). k_freq <= 8 runs the min/max network, 9 the selection passes."""
    L, E, d, N = 2, 64, 128, 2000
    Wr = torch.stack([synth.router_weights(E, d, 8, seed=40 + l) for l in range(L)])
    Wr[:, 10:14] = Wr[:, 9:10]          # five equal rows
    Wr[:, 40] = Wr[:, 20]
    Wr[:, 63] = Wr[:, 0]
    Wr = Wr.to(DEV).contiguous()
    Xcal = synth.calibration(N, d, seed=kf).to(DEV)
    ws = torch.empty(B.ordermoe_similarity_workspace_bytes(L, E, N), dtype=torch.uint8, device=DEV)
    sim = torch.empty(L, E, E, dtype=torch.float32, device=DEV)
    cnt = torch.empty(L, E, dtype=torch.int32, device=DEV)
    B.ordermoe_similarity(Wr, Xcal, L, E, d, N, kf, sim, cnt, ws)
    torch.cuda.synchronize()
    logits = ws[: N * L * E * 4].view(torch.float32).view(N, L * E).cpu().numpy()
    got = cnt.cpu().numpy()
    for l in range(L):
        lg = np.ascontiguousarray(logits[:, l * E:(l + 1) * E])
        assert (lg[:, 10] == lg[:, 9]).all() and (lg[:, 40] == lg[:, 20]).all()
        np.testing.assert_array_equal(got[l], oracle.expert_counts(lg, kf), err_msg="layer %d" % l)
        assert got[l].sum() == N * kf


def test_expert_counts_given_logits_bit_exact():
    rng = np.random.default_rng(3)
    for N, E, kf in [(5000, 64, 6), (100, 8, 2), (33, 5, 5)]:
        logits = rng.standard_normal((N, E)).astype(np.float32)
        logits[:10] = 0.5        # ties
        c = torch.empty(E, dtype=torch.int32, device=DEV)
        B.ordermoe_expert_counts(torch.as_tensor(logits).to(DEV), N, E, kf, c)
        np.testing.assert_array_equal(c.cpu().numpy(), oracle.expert_counts(logits, kf))


def gpu_place(sim, counts, M, p, C, theta_min=0.5, theta_max=0.9, theta_single=0.5):
    L, E, _ = sim.shape
    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a)).to(device=DEV, dtype=dt)
    group = torch.empty(L, E, dtype=torch.int32, device=DEV)
    ng = torch.empty(L, dtype=torch.int32, device=DEV)
    theta = torch.empty(L, dtype=torch.float32, device=DEV)
    x = torch.empty(L, M, E, dtype=torch.uint8, device=DEV)
    used = torch.empty(M, dtype=torch.float64, device=DEV)
    st = torch.empty(1, dtype=torch.int32, device=DEV)
    B.ordermoe_place(t(sim, torch.float32), t(counts, torch.int32), L, E, M, theta_min, theta_max,
                     theta_single, 0.5, 0.5, 0.5, 0.5, t(p, torch.float64), t(C, torch.float64),
                     group, ng, theta, None, x, used, st)
    torch.cuda.synchronize()
    return (group.cpu().numpy(), ng.cpu().numpy(), theta.cpu().numpy(), x.cpu().numpy(),
            used.cpu().numpy(), int(st.item()))


def oracle_place_all(sim, counts, M, p, C, theta_min=0.5, theta_max=0.9, theta_single=0.5):
    L, E, _ = sim.shape
    groups, ngs, thetas, imps = [], [], [], []
    for l in range(L):
        th = oracle.theta(l + 1, L, theta_min, theta_max, theta_single)
        g, K, _ = oracle.group(sim[l], counts[l], th)
        groups.append(g); ngs.append(K); thetas.append(th)
        imps.append(oracle.importance(sim[l], counts[l], g))
    x, used, rc = oracle.place(np.stack(groups), np.stack(imps), p, C)
    return np.stack(groups), np.array(ngs), np.array(thetas, np.float32), x, used, rc


def synthetic_sims(rng, L, E, K, noise):
    sims, counts = [], []
    for l in range(L):
        cen = rng.standard_normal((K, 32))
        Wt = cen[np.arange(E) % K] + noise * rng.standard_normal((E, 32))
        Wt /= np.linalg.norm(Wt, axis=1, keepdims=True)
        s = (Wt @ Wt.T).astype(np.float32)
        np.fill_diagonal(s, 1.0)
        sims.append(s)
        counts.append(rng.integers(0, 50, E).astype(np.int32))
    return np.stack(sims), np.stack(counts)


@pytest.mark.parametrize("L,E,M,K,noise", [(24, 64, 8, 8, 0.3), (1, 8, 4, 2, 0.25), (5, 16, 3, 4, 1.0),
                                           (32, 8, 4, 4, 0.25)])
def test_place_bit_exact(L, E, M, K, noise):
    rng = np.random.default_rng(L * E + M)
    sim, counts = synthetic_sims(rng, L, E, K, noise)
    p = np.ones((L, E)); C = np.full(M, L * E / M)
    got = gpu_place(sim, counts, M, p, C)
    ref = oracle_place_all(sim, counts, M, p, C)
    for name, a, b in zip(("group", "n_groups", "theta", "placement", "used", "status"), got, ref):
        np.testing.assert_array_equal(a, b, err_msg=name)


@pytest.mark.parametrize("L,E,M,scale,frac", [(4, 1, 2, 1.0, False), (5, 2, 3, 1.2, True),
                                                (6, 3, 2, 0.9, False), (9, 64, 16, 1.1, False),
                                                (9, 64, 17, 1.1, True), (12, 37, 16, 0.95, True),
                                                (3, 40, 1, 1.0, False), (20, 24, 7, 0.97, False)])
def test_place_ties_waiting_lists_and_server_counts(L, E, M, scale, frac):
    """Integer sizes and equal capacities give exact score ties (to the lower
    server); capacities below the demand send experts to the waiting list and
    report the overflow; one to 17 servers, one to 64 experts a layer."""
    rng = np.random.default_rng(L * 1000 + E * 10 + M)
    sim, counts = synthetic_sims(rng, L, E, max(1, min(4, E)), 0.4)
    if frac:
        p = rng.uniform(0.5, 2.5, (L, E)); C = p.sum() / M * scale * rng.uniform(0.9, 1.1, M)
    else:
        p = rng.integers(1, 4, (L, E)).astype(np.float64); C = np.full(M, np.ceil(p.sum() / M * scale))
    got = gpu_place(sim, counts, M, p, C)
    ref = oracle_place_all(sim, counts, M, p, C)
    for name, a, b in zip(("group", "n_groups", "theta", "placement", "used", "status"), got, ref):
        np.testing.assert_array_equal(a, b, err_msg="%s L=%d E=%d M=%d" % (name, L, E, M))
    assert (got[3].sum(axis=1) == 1).all()  # every expert on exactly one server


@pytest.mark.parametrize("E", [64, 40, 8])
def test_group_exact_ties_and_signed_zeros_match_oracle(E):
    """Similarities drawn from a few exact values give an expert several
    equally similar dominants (Eqs. 24-26: the scan keeps the lowest
    dominant); in the last layer (threshold -0.25) the only values are +0, -0
    and -0.5, so the most similar dominants tie at zero of either sign, which
    compare equal. Counts tie too (the visiting order: count desc, index asc).
    Groups, group counts, thresholds and placements bit for bit."""
    rng = np.random.default_rng(700 + E)
    L, M = 4, 8
    sets = [np.array([0.95, 0.95, 0.3, 0.0, -0.0, -0.5], np.float32)] * (L - 1) + \
        [np.array([0.0, -0.0, -0.5], np.float32)]
    sims = []
    for l in range(L):
        u = rng.choice(sets[l], (E, E)).astype(np.float32)
        # symmetric by mirroring the upper triangle (a sum would turn -0 into +0)
        s = np.where(np.triu(np.ones((E, E), bool), 1), u, u.T).astype(np.float32)
        np.fill_diagonal(s, 1.0)
        sims.append(s)
    sim = np.stack(sims)
    assert np.signbit(sim[L - 1][sim[L - 1] == 0]).any()   # both signs of zero present
    counts = rng.integers(0, 4, (L, E)).astype(np.int32)
    p = np.ones((L, E)); C = np.full(M, L * E / M * 1.5)
    got = gpu_place(sim, counts, M, p, C, theta_min=-0.25, theta_max=0.9)
    ref = oracle_place_all(sim, counts, M, p, C, theta_min=-0.25, theta_max=0.9)
    for name, a, b in zip(("group", "n_groups", "theta", "placement", "used", "status"), got, ref):
        np.testing.assert_array_equal(a, b, err_msg="%s E=%d" % (name, E))
    assert ref[1][L - 1] < E                                  # experts joined dominants at zero


def test_place_with_nan_similarities_matches_oracle():
    """NaN similarities (bad inputs) give the oracle's groups, importances
    (NaN where a group mean meets one), placement order and placement: the
    grouping follows the scan's rule, and NaN importances go after every
    number."""
    rng = np.random.default_rng(31)
    L, E, M = 6, 16, 4
    sim, counts = synthetic_sims(rng, L, E, 4, 0.4)
    for l in range(L):
        for _ in range(3):  # symmetric NaN pairs off the diagonal
            i, j = rng.choice(E, 2, replace=False)
            sim[l, i, j] = sim[l, j, i] = np.nan
    # a NaN to the first dominant (the expert with the most activations)
    first = int(np.argmax(counts[0])); other = (first + 1) % E
    sim[0, first, other] = sim[0, other, first] = np.nan
    p = np.ones((L, E)); C = np.full(M, L * E / M * 1.2)
    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a)).to(device=DEV, dtype=dt)
    group = torch.empty(L, E, dtype=torch.int32, device=DEV)
    ng = torch.empty(L, dtype=torch.int32, device=DEV)
    theta = torch.empty(L, dtype=torch.float32, device=DEV)
    imp = torch.empty(L, E, dtype=torch.float64, device=DEV)
    x = torch.empty(L, M, E, dtype=torch.uint8, device=DEV)
    used = torch.empty(M, dtype=torch.float64, device=DEV)
    st = torch.empty(1, dtype=torch.int32, device=DEV)
    B.ordermoe_place(t(sim, torch.float32), t(counts, torch.int32), L, E, M, 0.5, 0.9, 0.5, 0.5, 0.5,
                     0.5, 0.5, t(p, torch.float64), t(C, torch.float64), group, ng, theta, imp, x, used, st)
    torch.cuda.synchronize()
    ref = oracle_place_all(sim, counts, M, p, C)
    got = (group.cpu().numpy(), ng.cpu().numpy(), theta.cpu().numpy(), x.cpu().numpy(),
           used.cpu().numpy(), int(st.item()))
    for name, a, b in zip(("group", "n_groups", "theta", "placement", "used", "status"), got, ref):
        np.testing.assert_array_equal(a, b, err_msg=name)
    ref_imp = np.stack([oracle.importance(sim[l], counts[l], ref[0][l]) for l in range(L)])
    np.testing.assert_array_equal(imp.cpu().numpy(), ref_imp)
    assert np.isnan(ref_imp).any()
    assert (got[3].sum(axis=1) == 1).all()


def test_place_reports_a_bad_memory_demand():
    """A negative or NaN memory demand p is reported (ORDERMOE_DEV_BAD_VALUE,
    detail = l * E + j) and the call still completes."""
    rng = np.random.default_rng(41)
    L, E, M = 3, 8, 2
    sim, counts = synthetic_sims(rng, L, E, 2, 0.4)
    for bad, where in ((np.nan, (1, 5)), (-1.0, (2, 0))):
        p = np.ones((L, E)); p[where] = bad
        gpu_place(sim, counts, M, p, np.full(M, L * E))
        code, detail = B.ordermoe_device_error()
        assert code == B.DEV_BAD_VALUE and detail == where[0] * E + where[1], (bad, code, detail)
    gpu_place(sim, counts, M, np.ones((L, E)), np.full(M, L * E))
    assert B.ordermoe_device_error()[0] == 0


def test_placement_quotient_is_correctly_rounded():
    """The placement's load ratio b_m / C_m (reciprocal + Markstein's correction)
    equals IEEE division (numpy) bit for bit on random and edge operands."""
    rng = np.random.default_rng(17)
    n = 1 << 22
    a = np.concatenate([rng.random(n // 4) * 1e3, np.floor(rng.random(n // 4) * 4096),
                        2.0 ** rng.uniform(-300, 300, n // 4) * rng.uniform(1, 2, n // 4),
                        rng.integers(0, 1 << 40, n // 4).astype(np.float64)])
    b = np.concatenate([rng.random(n // 4) * 1e3 + 1e-3, np.floor(rng.random(n // 4) * 512) + 1,
                        2.0 ** rng.uniform(-300, 300, n // 4) * rng.uniform(1, 2, n // 4),
                        rng.integers(1, 1 << 30, n // 4).astype(np.float64)])
    b[:64] = 1.0; a[64:128] = 0.0; b[128:192] = 3.0; a[128:192] = np.arange(64)   # exact and repeating
    bits = rng.integers(0, 1 << 52, 2 * 4096, dtype=np.int64)
    a[192:4288] = (bits[:4096] | (1023 << 52)).view(np.float64)                    # [1, 2) all mantissas
    b[192:4288] = (bits[4096:] | (1023 << 52)).view(np.float64)
    out = torch.empty(n, dtype=torch.float64, device=DEV)
    B.ordermoe_selftest_div_rn(torch.as_tensor(a).to(DEV), torch.as_tensor(b).to(DEV), out)
    got = out.cpu().numpy()
    want = a / b
    bad = np.nonzero(got.view(np.int64) != want.view(np.int64))[0]
    assert bad.size == 0, (bad[:5], a[bad[:5]], b[bad[:5]], got[bad[:5]], want[bad[:5]])


def test_place_fractional_sizes_and_capacities_bit_exact():
    rng = np.random.default_rng(23)
    for L, E, M in [(40, 64, 32), (7, 13, 5), (64, 8, 3)]:
        sim, counts = synthetic_sims(rng, L, E, 4, 0.4)
        p = rng.uniform(0.5, 2.5, (L, E))
        C = p.sum() / M * rng.uniform(1.05, 1.6, M)
        got = gpu_place(sim, counts, M, p, C)
        ref = oracle_place_all(sim, counts, M, p, C)
        for name, a, b in zip(("group", "n_groups", "theta", "placement", "used", "status"), got, ref):
            np.testing.assert_array_equal(a, b, err_msg="%s L=%d E=%d M=%d" % (name, L, E, M))


def test_place_unequal_sizes_waiting_list_and_capacity():
    rng = np.random.default_rng(9)
    L, E, M = 3, 6, 3
    sim, counts = synthetic_sims(rng, L, E, 2, 0.5)
    p = rng.integers(1, 4, (L, E)).astype(np.float64)
    for scale in (1.0, 0.9, 1.3):
        C = np.full(M, p.sum() / M * scale)
        got = gpu_place(sim, counts, M, p, C)
        ref = oracle_place_all(sim, counts, M, p, C)
        for name, a, b in zip(("group", "n_groups", "theta", "placement", "used", "status"), got, ref):
            np.testing.assert_array_equal(a, b, err_msg="%s scale %g" % (name, scale))


def gpu_replicate(group, I, p, C, pi, x, used):
    L, E = group.shape; M = len(C)
    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a)).to(device=DEV, dtype=dt)
    gx = t(x, torch.uint8); gb = t(used, torch.float64)
    reps = torch.empty(M, dtype=torch.int32, device=DEV)
    B.ordermoe_replicate(t(group, torch.int32), t(I, torch.float64), t(p, torch.float64),
                         t(C, torch.float64), t(pi, torch.float64), L, E, M, gx, gb, reps)
    torch.cuda.synchronize()
    return gx.cpu().numpy(), gb.cpu().numpy(), reps.cpu().numpy()


def test_place_importance_output_bit_exact():
    rng = np.random.default_rng(2)
    L, E, M = 6, 16, 4
    sim, counts = synthetic_sims(rng, L, E, 4, 0.4)
    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a)).to(device=DEV, dtype=dt)
    group = torch.empty(L, E, dtype=torch.int32, device=DEV)
    imp = torch.empty(L, E, dtype=torch.float64, device=DEV)
    x = torch.empty(L, M, E, dtype=torch.uint8, device=DEV)
    B.ordermoe_place(t(sim, torch.float32), t(counts, torch.int32), L, E, M, 0.5, 0.9, 0.5, 0.5, 0.5,
                     0.5, 0.5, t(np.ones((L, E)), torch.float64), t(np.full(M, L * E / M), torch.float64),
                     group, torch.empty(L, dtype=torch.int32, device=DEV),
                     torch.empty(L, dtype=torch.float32, device=DEV), imp, x,
                     torch.empty(M, dtype=torch.float64, device=DEV),
                     torch.empty(1, dtype=torch.int32, device=DEV))
    g = group.cpu().numpy()
    for l in range(L):
        np.testing.assert_array_equal(imp[l].cpu().numpy(), oracle.importance(sim[l], counts[l], g[l]))


@pytest.mark.parametrize("L,E,M,ratio,seed", [(1, 4, 2, 1.5, 0), (3, 6, 3, 2.0, 1), (5, 16, 5, 1.3, 2),
                                              (7, 13, 6, 2.5, 3), (32, 8, 8, 2.0, 4), (24, 64, 8, 2.0, 5),
                                              (2, 64, 32, 3.0, 6)])
def test_replicate_bit_exact(L, E, M, ratio, seed):
    """Redundant deployment after the mandatory placement, unequal memory
    demands, ties and non-positive importances, servers no token reaches."""
    rng = np.random.default_rng(seed)
    K = max(1, E // 4)
    group = rng.integers(0, K, (L, E)).astype(np.int32)
    I = rng.random((L, E)); I[rng.random((L, E)) < 0.15] = 0.5; I[rng.random((L, E)) < 0.05] = -0.1
    p = rng.integers(1, 4, (L, E)).astype(np.float64) if seed % 2 else np.ones((L, E))
    C = synth.capacities(M, p.sum(), ratio, seed)
    x0, used0, rc = oracle.place(group, np.abs(I), p, C)
    assert rc == 0
    pi = synth.token_shares(synth.homes(4096, M, seed, "zipf1.1"), M)
    pi[rng.random(M) < 0.2] = 0.0
    ref = oracle.replicate(group, I, p, C, pi, x0, used0)
    got = gpu_replicate(group, I, p, C, pi, x0, used0)
    for name, a, b in zip(("placement", "used", "replicas"), got, ref):
        np.testing.assert_array_equal(a, b, err_msg=name)
    if L * E >= 64:
        assert ref[2].sum() > 0


def test_replicate_largest_shape_and_errors():
    rng = np.random.default_rng(8)
    L, E, M = 256, 64, 4                          # L * E = 16384, the largest sort
    group = rng.integers(0, 16, (L, E)).astype(np.int32)
    I = rng.random((L, E)); p = np.ones((L, E))
    C = np.full(M, L * E / M * 1.05)
    x0, used0, rc = oracle.place(group, I, p, C)
    assert rc == 0
    pi = np.array([0.4, 0.3, 0.2, 0.1])
    ref = oracle.replicate(group, I, p, C, pi, x0, used0)
    got = gpu_replicate(group, I, p, C, pi, x0, used0)
    for name, a, b in zip(("placement", "used", "replicas"), got, ref):
        np.testing.assert_array_equal(a, b, err_msg=name)
    # the most layers (1024), unequal memory demands
    L2, E2, M2 = 1024, 16, 3
    group2 = rng.integers(0, 4, (L2, E2)).astype(np.int32)
    I2 = rng.random((L2, E2)); p2 = rng.integers(1, 4, (L2, E2)).astype(np.float64)
    C2 = np.full(M2, p2.sum() / M2 * 1.1)
    x2, used2, rc = oracle.place(group2, I2, p2, C2)
    assert rc == 0
    pi2 = np.array([0.5, 0.3, 0.2])
    ref = oracle.replicate(group2, I2, p2, C2, pi2, x2, used2)
    got = gpu_replicate(group2, I2, p2, C2, pi2, x2, used2)
    for name, a, b in zip(("placement", "used", "replicas"), got, ref):
        np.testing.assert_array_equal(a, b, err_msg="L 1024 " + name)
    assert ref[2].min() > 0
    with pytest.raises(B.OrderMoEError) as ei:
        gpu_replicate(np.zeros((257, 64), np.int32), np.ones((257, 64)), np.ones((257, 64)), C, pi,
                      np.zeros((257, 4, 64), np.uint8), np.zeros(4))
    assert ei.value.code == B.ERR_UNSUPPORTED_SHAPE
    # a non-positive memory demand is reported and skipped
    p_bad = np.ones((1, 4)); p_bad[0, 2] = 0.0
    gpu_replicate(np.array([[0, 0, 1, 1]], np.int32), np.ones((1, 4)), p_bad, np.array([9.0, 9.0]),
                  np.array([0.5, 0.5]), np.zeros((1, 2, 4), np.uint8), np.zeros(2))
    code, detail = B.ordermoe_device_error()
    assert code == B.DEV_BAD_VALUE and detail == 2


@pytest.mark.parametrize("L,E,M", [(1, 4, 2), (24, 64, 8), (32, 8, 8), (3, 64, 32), (5, 48, 6), (4, 40, 3)])
def test_coverage_bit_exact(L, E, M):
    rng = np.random.default_rng(L + E + M)
    group = rng.integers(0, max(1, E // 3), (L, E)).astype(np.int32)
    x = (rng.random((L, M, E)) < 0.2).astype(np.uint8)
    gc = torch.empty(L, M, E, dtype=torch.uint8, device=DEV)
    gn = torch.empty(L, dtype=torch.int32, device=DEV)
    B.ordermoe_coverage(torch.as_tensor(group).to(DEV), torch.as_tensor(x).to(DEV), L, E, M, gc, gn)
    cov = gc.cpu().numpy()
    for l in range(L):
        ref = oracle.coverage(x[l], group[l], E)
        np.testing.assert_array_equal(cov[l], ref)
        assert gn[l].item() == int(ref.sum())


def test_redundant_plan_at_memory_ratio_two_raises_coverage():
    """The whole of Alg. 1 on the GPU for 32 Mixtral-shaped layers, 8 servers:
    placement, then redundancy at memory ratio 2.0 with pi from Zipf homes;
    coverage goes up and matches the oracle's plan."""
    rng = np.random.default_rng(12)
    L, E, M = 32, 8, 8
    sim, counts = synthetic_sims(rng, L, E, 4, 0.3)
    p = np.ones((L, E)); C = synth.capacities(M, L * E, 2.0, 12)
    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a)).to(device=DEV, dtype=dt)
    group = torch.empty(L, E, dtype=torch.int32, device=DEV)
    ng = torch.empty(L, dtype=torch.int32, device=DEV)
    imp = torch.empty(L, E, dtype=torch.float64, device=DEV)
    x = torch.empty(L, M, E, dtype=torch.uint8, device=DEV)
    used = torch.empty(M, dtype=torch.float64, device=DEV)
    st = torch.empty(1, dtype=torch.int32, device=DEV)
    gp, gC = t(p, torch.float64), t(C, torch.float64)
    B.ordermoe_place(t(sim, torch.float32), t(counts, torch.int32), L, E, M, 0.5, 0.9, 0.5, 0.5, 0.5,
                     0.5, 0.5, gp, gC, group, ng, torch.empty(L, dtype=torch.float32, device=DEV), imp,
                     x, used, st)
    covered0 = torch.empty(L, dtype=torch.int32, device=DEV)
    B.ordermoe_coverage(group, x, L, E, M, None, covered0)
    x0, used0 = x.cpu().numpy(), used.cpu().numpy()
    pi = synth.token_shares(synth.homes(8192, M, 12, "zipf1.1"), M)
    reps = torch.empty(M, dtype=torch.int32, device=DEV)
    B.ordermoe_replicate(group, imp, gp, gC, t(pi, torch.float64), L, E, M, x, used, reps)
    covered = torch.empty(L, dtype=torch.int32, device=DEV)
    B.ordermoe_coverage(group, x, L, E, M, None, covered)
    total = M * int(ng.sum().item())
    before, after = covered0.sum().item() / total, covered.sum().item() / total
    print("local group coverage: %.3f -> %.3f with %d replicas" % (before, after, int(reps.sum().item())))
    assert st.item() == 0 and after > before
    assert (used.cpu().numpy() <= C).all()
    ref = oracle.replicate(group.cpu().numpy(), imp.cpu().numpy(), p, C, pi, x0, used0)
    np.testing.assert_array_equal(x.cpu().numpy(), ref[0])
    np.testing.assert_array_equal(reps.cpu().numpy(), ref[2])


def test_similarity_full_size():
    """The similarity workload at full size: 24 layers x 64 clustered experts,
    d = 2048, N = 262144 calibration tokens (Eqs. 3-5), then Alg. 1 on the
    GPU's own similarities and counts (Eqs. 24-35).
    - Eq. 3: the GPU's fp32 calibration logits on 512 sampled tokens of two
      layers against the oracle's fp64 sums;
    - Eq. 5: the counts of every layer recomputed by the oracle from the GPU's
      own fp32 logits, bit for bit (the same top-k and tie rule on the same
      inputs);
    - Eq. 4: one whole 64 x 64 layer of Sim against the fp64 oracle within
      2e-5, and sampled expert pairs of two more layers;
    - Eqs. 24-31: grouping, theta_l, importance and placement of every layer,
      and (Eqs. 32-35) the replicas and local group coverage at memory ratio
      2.0, each from the oracle run on the GPU's similarities and counts, bit
      for bit;
    - properties at any size: symmetry, |Sim| <= 1, counts summing to N k, the
      8 router clusters recovered as groups, c.1 and c.2."""
    w = synth.workload("similarity")
    L, E, d, N, M, kf = w.L, w.E, w.d, w.n_cal, w.M, w.k
    Wr = torch.stack([synth.router_weights(E, d, w.n_clusters, seed=500 + l, device=DEV)
                      for l in range(L)])
    Xcal = synth.calibration(N, d, seed=1, device=DEV)
    sim_t = torch.empty(L, E, E, dtype=torch.float32, device=DEV)
    counts_t = torch.empty(L, E, dtype=torch.int32, device=DEV)
    ws = torch.empty(B.ordermoe_similarity_workspace_bytes(L, E, N), dtype=torch.uint8, device=DEV)
    B.ordermoe_similarity(Wr, Xcal, L, E, d, N, kf, sim_t, counts_t, ws)
    torch.cuda.synchronize()
    sim, counts = sim_t.cpu().numpy(), counts_t.cpu().numpy()
    logits = ws[:N * L * E * 4].view(torch.float32).view(N, L, E).cpu().numpy()
    del ws
    assert np.allclose(sim, np.transpose(sim, (0, 2, 1)), atol=1e-6)
    assert (np.abs(sim) <= 1 + 1e-6).all()
    assert (counts.sum(axis=1) == N * kf).all()
    rng = np.random.default_rng(0)
    Xb = synth.bits(Xcal)
    tok = np.sort(rng.choice(N, 512, replace=False))
    for l in (0, 23):
        ref = oracle.router_logits(Xb[tok], synth.bits(Wr[l]))
        np.testing.assert_allclose(logits[tok, l, :], ref, rtol=1e-3, atol=2e-3)
    for l in range(L):
        ref = oracle.expert_counts(np.ascontiguousarray(logits[:, l, :]), kf)
        np.testing.assert_array_equal(counts[l], ref, err_msg="counts of layer %d" % l)
    del logits
    np.testing.assert_allclose(sim[7], oracle.similarity(synth.bits(Wr[7]), Xb), atol=2e-5)
    for l in (0, 23):
        ex = np.sort(rng.choice(E, 3, replace=False))
        ref = oracle.similarity(synth.bits(Wr[l][ex]), Xb)
        np.testing.assert_allclose(sim[l][np.ix_(ex, ex)], ref, atol=2e-5)
    # Alg. 1 on the GPU's similarities and counts, at memory ratio 2.0
    p = np.ones((L, E)); C = synth.capacities(M, L * E, 2.0, 3)
    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a)).to(device=DEV, dtype=dt)
    group = torch.empty(L, E, dtype=torch.int32, device=DEV)
    ng = torch.empty(L, dtype=torch.int32, device=DEV)
    theta = torch.empty(L, dtype=torch.float32, device=DEV)
    imp = torch.empty(L, E, dtype=torch.float64, device=DEV)
    x = torch.empty(L, M, E, dtype=torch.uint8, device=DEV)
    used = torch.empty(M, dtype=torch.float64, device=DEV)
    st = torch.empty(1, dtype=torch.int32, device=DEV)
    gp, gC = t(p, torch.float64), t(C, torch.float64)
    B.ordermoe_place(sim_t, counts_t, L, E, M, w.theta_min, w.theta_max, w.theta, 0.5, 0.5, 0.5,
                     0.5, gp, gC, group, ng, theta, imp, x, used, st)
    torch.cuda.synchronize()
    got = (group.cpu().numpy(), ng.cpu().numpy(), theta.cpu().numpy(), x.cpu().numpy(),
           used.cpu().numpy(), int(st.item()))
    ref = oracle_place_all(sim, counts, M, p, C, w.theta_min, w.theta_max, w.theta)
    for name, a, b in zip(("group", "n_groups", "theta", "placement", "used", "status"), got, ref):
        np.testing.assert_array_equal(a, b, err_msg=name)
    ref_imp = np.stack([oracle.importance(sim[l], counts[l], ref[0][l]) for l in range(L)])
    np.testing.assert_array_equal(imp.cpu().numpy(), ref_imp)
    pi = synth.token_shares(synth.homes(8192, M, 3, "zipf1.1"), M)
    reps = torch.empty(M, dtype=torch.int32, device=DEV)
    B.ordermoe_replicate(group, imp, gp, gC, t(pi, torch.float64), L, E, M, x, used, reps)
    cov = torch.empty(L, M, E, dtype=torch.uint8, device=DEV)
    covered = torch.empty(L, dtype=torch.int32, device=DEV)
    B.ordermoe_coverage(group, x, L, E, M, cov, covered)
    torch.cuda.synchronize()
    rx, rused, rreps = oracle.replicate(ref[0], ref_imp, p, C, pi, ref[3], ref[4])
    np.testing.assert_array_equal(x.cpu().numpy(), rx)
    np.testing.assert_array_equal(used.cpu().numpy(), rused)
    np.testing.assert_array_equal(reps.cpu().numpy(), rreps)
    gcov = cov.cpu().numpy()
    for l in range(L):
        rc = oracle.coverage(rx[l], ref[0][l], E)
        np.testing.assert_array_equal(gcov[l], rc, err_msg="coverage of layer %d" % l)
        assert covered[l].item() == int(rc.sum())
    # what the workload is built to show: the 8 router clusters (cosine ~0.94
    # inside a cluster, ~0 across, against theta_l in [0.5, 0.9]) become the
    # groups, every expert placed once (c.2), no server over capacity (c.1)
    gr = ref[0]
    assert ref[5] == 0 and (ref[1] == w.n_clusters).all()
    cl = synth.cluster_of(E, w.n_clusters)
    for l in range(L):
        np.testing.assert_array_equal(gr[l][:, None] == gr[l][None, :], cl[:, None] == cl[None, :])
    assert (ref[3].sum(axis=1) == 1).all()
    assert (rused <= C + 1e-9).all()


# ------------------------------------------------------------------ whole-layer entry

def test_layer_forward_device_and_host_io_match_the_stepwise_path():
    from paper_2607_17154_gb300.layer import MoELayer
    from tests.helpers import oracle_plan
    w = synth.workload("tiny", T=200)
    inp = synth.layer_inputs(w, seed=4)
    plan = oracle_plan(synth.bits(inp["Wr"]), synth.bits(synth.calibration(w.n_cal, w.d, 4)),
                       w.k, w.M, w.theta)
    sp = synth.server_params(w.M, w.d, w.dff, 4)
    tab = build_tables(plan["sim"], plan["group"], plan["placement"], w.theta, w.qbar, sp, DEV)
    g = {n: inp[n].to(DEV) for n in ("X", "Wr", "W1", "W3", "W2")}
    home = torch.as_tensor(inp["home"]).to(DEV)
    layer = MoELayer(g["Wr"], g["W1"], g["W3"], g["W2"], tab, w.k, w.T)
    y_ref = torch.empty(w.T, w.d, dtype=torch.bfloat16, device=DEV)
    layer.forward(g["X"], home, home.clone(), torch.zeros(w.T, device=DEV), y_ref)
    scratch = torch.empty(B.ordermoe_layer_scratch_bytes(256, w.E, w.d, w.dff, w.k),
                          dtype=torch.uint8, device=DEV)
    desc = B.make_layer_desc(256, g["Wr"], g["W1"], g["W3"], g["W2"], tab, w.k, scratch)
    y_dev = torch.empty(w.T, w.d, dtype=torch.bfloat16, device=DEV)
    B.ordermoe_layer_forward(desc, w.T, g["X"], home, None, None, y_dev)
    Xh = inp["X"].pin_memory(); hh = torch.as_tensor(inp["home"]).pin_memory()
    yh = torch.empty(w.T, w.d, dtype=torch.bfloat16).pin_memory()
    loch = hh.clone(); qh = torch.zeros(w.T).pin_memory()
    B.ordermoe_layer_forward(desc, w.T, Xh, hh, loch, qh, yh, host_io=1)
    torch.cuda.synchronize()
    assert torch.equal(y_dev.cpu(), y_ref.cpu())
    assert torch.equal(yh, y_ref.cpu())
    assert torch.equal(loch, torch.as_tensor(layer.server[:, 0].cpu()))
    # deterministic: a second call gives the same bits
    y2 = torch.empty_like(y_dev)
    B.ordermoe_layer_forward(desc, w.T, g["X"], home, None, None, y2)
    torch.cuda.synchronize()
    assert torch.equal(y2, y_dev)


def test_layer_forward_batches_matches_single_calls():
    """Five batches through the overlapped host-I/O entry point (both staging
    slots reused) give each batch's single-call output bit for bit, and the
    execution-type counters add up."""
    w = synth.workload("tiny")
    E, d, dff, k, M = w.E, w.d, w.dff, w.k, w.M
    T, nb = 200, 5
    inp = synth.layer_inputs(w, seed=3, device=DEV)
    rng = np.random.default_rng(3)
    sim, group, x = random_tables_case(rng, E, M, 2)
    tab = build_tables(sim, group, x, 0.5, w.qbar, synth.server_params(M, d, dff, 0), DEV)
    scratch = torch.empty(B.ordermoe_layer_batches_scratch_bytes(T, E, d, dff, k), dtype=torch.uint8,
                          device=DEV)
    desc = B.make_layer_desc(T, inp["Wr"], inp["W1"], inp["W3"], inp["W2"], tab, k, scratch)
    X = torch.stack([synth.hidden(T, d, 40 + b) for b in range(nb)]).pin_memory()
    home = torch.as_tensor(rng.integers(0, M, (nb, T)).astype(np.uint8)).pin_memory()
    y = torch.zeros(nb, T, d, dtype=torch.bfloat16).pin_memory()
    cnt = torch.zeros(4, dtype=torch.int32, device=DEV)
    B.ordermoe_layer_forward_batches(desc, nb, T, X, home, y, cnt)
    torch.cuda.synchronize()
    assert cnt.sum().item() == nb * T * k
    for b in range(nb):
        y1 = torch.zeros(T, d, dtype=torch.bfloat16).pin_memory()
        B.ordermoe_layer_forward(desc, T, X[b], home[b], None, None, y1, host_io=1)
        torch.cuda.synchronize()
        assert torch.equal(y[b], y1), b


def test_layer_forward_batches_from_two_host_threads():
    """Two host threads, each with its own layer scratch and stream, run the
    batched host-I/O entry point at the same time (the device's copy streams
    and events are shared): each gets its single-call outputs."""
    import threading
    w = synth.workload("tiny")
    E, d, dff, k, M = w.E, w.d, w.dff, w.k, w.M
    T, nb = 128, 4
    inp = synth.layer_inputs(w, seed=5, device=DEV)
    rng = np.random.default_rng(5)
    sim, group, x = random_tables_case(rng, E, M, 2)
    tab = build_tables(sim, group, x, 0.5, w.qbar, synth.server_params(M, d, dff, 0), DEV)
    jobs = []
    for i in range(2):
        scratch = torch.empty(B.ordermoe_layer_batches_scratch_bytes(T, E, d, dff, k), dtype=torch.uint8,
                              device=DEV)
        desc = B.make_layer_desc(T, inp["Wr"], inp["W1"], inp["W3"], inp["W2"], tab, k, scratch)
        X = torch.stack([synth.hidden(T, d, 80 + 10 * i + b) for b in range(nb)]).pin_memory()
        home = torch.as_tensor(rng.integers(0, M, (nb, T)).astype(np.uint8)).pin_memory()
        ref = []
        for b in range(nb):
            y1 = torch.zeros(T, d, dtype=torch.bfloat16).pin_memory()
            B.ordermoe_layer_forward(desc, T, X[b], home[b], None, None, y1, host_io=1)
            ref.append(y1)
        jobs.append((desc, scratch, X, home, ref))
    torch.cuda.synchronize()
    outs = [[], []]
    errors = []

    def run(i):
        try:
            desc, _, X, home, _ = jobs[i]
            s = torch.cuda.Stream()
            with torch.cuda.stream(s):
                for _ in range(3):
                    y = torch.zeros(nb, T, d, dtype=torch.bfloat16).pin_memory()
                    B.ordermoe_layer_forward_batches(desc, nb, T, X, home, y, None)
                    outs[i].append(y)
            s.synchronize()
        except Exception as e:  # reported below, in the test's thread
            errors.append(e)

    threads = [threading.Thread(target=run, args=(i,)) for i in range(2)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    torch.cuda.synchronize()
    assert not errors, errors
    for i in range(2):
        assert len(outs[i]) == 3
        for y in outs[i]:
            for b in range(nb):
                assert torch.equal(y[b], jobs[i][4][b]), (i, b)


def _plan_inputs(L, E, d, N, M, seed, unequal):
    Wr = torch.stack([synth.router_weights(E, d, 4, seed=seed + 70 + l) for l in range(L)]).to(DEV).contiguous()
    Xcal = synth.calibration(N, d, seed=seed + 3).to(DEV)
    rng = np.random.default_rng(seed)
    p = rng.integers(1, 4, (L, E)).astype(np.float64) if unequal else np.ones((L, E))
    C = synth.capacities(M, p.sum(), 1.6, seed)
    pi = synth.token_shares(synth.homes(4096, M, seed, "zipf1.1"), M)
    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a)).to(device=DEV, dtype=dt)
    return Wr, Xcal, t(p, torch.float64), t(C, torch.float64), t(pi, torch.float64)


def _plan_outputs(L, E, M):
    f = lambda *s, dt: torch.full(s, 7, dtype=dt, device=DEV)
    return dict(sim=f(L, E, E, dt=torch.float32), counts=f(L, E, dt=torch.int32),
                group=f(L, E, dt=torch.int32), n_groups=f(L, dt=torch.int32),
                theta=f(L, dt=torch.float32), importance=f(L, E, dt=torch.float64),
                placement=f(L, M, E, dt=torch.uint8), used=f(M, dt=torch.float64),
                status=f(1, dt=torch.int32), replicas=f(M, dt=torch.int32),
                cover=f(L, M, E, dt=torch.uint8), covered=f(L, dt=torch.int32))


TH = (0.5, 0.9, 0.6, 0.5, 0.5, 0.5, 0.5)  # theta_min, theta_max, theta_single, alpha_f, alpha_r, lambda1, lambda2


def _serial_plan(Wr, Xcal, L, E, d, N, kf, M, p, C, pi):
    o = _plan_outputs(L, E, M)
    ws = torch.empty(B.ordermoe_similarity_workspace_bytes(L, E, N), dtype=torch.uint8, device=DEV)
    B.ordermoe_similarity_no_logits(Wr, Xcal, L, E, d, N, kf, o["sim"], o["counts"], ws)
    B.ordermoe_place(o["sim"], o["counts"], L, E, M, *TH, p, C, o["group"], o["n_groups"], o["theta"],
                     o["importance"], o["placement"], o["used"], o["status"])
    B.ordermoe_replicate(o["group"], o["importance"], p, C, pi, L, E, M, o["placement"], o["used"],
                         o["replicas"])
    B.ordermoe_coverage(o["group"], o["placement"], L, E, M, o["cover"], o["covered"])
    return o


def _one_plan(Wr, Xcal, L, E, d, N, kf, M, p, C, pi, ws, stream=None):
    o = _plan_outputs(L, E, M)
    B.ordermoe_plan(Wr, Xcal, L, E, d, N, kf, M, *TH, p, C, pi, o["sim"], o["counts"], o["group"],
                    o["n_groups"], o["theta"], o["importance"], o["placement"], o["used"], o["status"],
                    o["replicas"], o["cover"], o["covered"], ws, stream=stream)
    return o


def _same(a, b, what):
    for k in a:
        assert torch.equal(a[k], b[k]), "%s: %s differs" % (what, k)


@pytest.mark.parametrize("L,E,N,M,kf,unequal", [(24, 64, 4096, 8, 6, False), (13, 64, 3000, 4, 6, True),
                                                 (1, 64, 1000, 3, 2, False), (20, 32, 2100, 5, 4, True),
                                                 (40, 16, 1500, 16, 3, False), (80, 8, 1200, 6, 2, True),
                                                 (3, 12, 900, 3, 3, False), (64, 64, 700, 8, 6, True),
                                                 (65, 64, 700, 8, 6, False)])
def test_plan_equals_the_four_calls(L, E, N, M, kf, unequal):
    """ordermoe_plan (blocks of 512 logit columns; grouping and placement of a
    block on a side stream while the next block's GEMM runs) writes what the
    four calls write one after the other, bit for bit: ragged last blocks,
    b_m carried across blocks, the tensor-core limit L E = 4096 (8 blocks),
    and the one-stream path for E = 12 and for L E = 4160."""
    d = 128
    Wr, Xcal, p, C, pi = _plan_inputs(L, E, d, N, M, L * 7 + E, unequal)
    ref = _serial_plan(Wr, Xcal, L, E, d, N, kf, M, p, C, pi)
    ws = torch.empty(B.ordermoe_plan_workspace_bytes(L, E, N), dtype=torch.uint8, device=DEV)
    got = _one_plan(Wr, Xcal, L, E, d, N, kf, M, p, C, pi, ws)
    torch.cuda.synchronize()
    _same(got, ref, "plan")
    assert int(ref["status"].item()) in (B.OK, B.ERR_CAPACITY)
    assert (got["placement"].sum(dim=1) >= 1).all()  # every expert somewhere


def test_plan_back_to_back_and_in_a_cuda_graph():
    """Calls queued back to back on one stream (the library's events reused)
    and a captured-and-replayed call give the single call's results; work
    queued after the call on the caller's stream sees its outputs."""
    L, E, d, N, M, kf = 13, 64, 128, 2000, 6, 6
    Wr, Xcal, p, C, pi = _plan_inputs(L, E, d, N, M, 5, True)
    ws = torch.empty(B.ordermoe_plan_workspace_bytes(L, E, N), dtype=torch.uint8, device=DEV)
    ref = _one_plan(Wr, Xcal, L, E, d, N, kf, M, p, C, pi, ws)
    torch.cuda.synchronize()
    runs = [_one_plan(Wr, Xcal, L, E, d, N, kf, M, p, C, pi, ws) for _ in range(3)]
    after = [r["placement"].to(torch.int32).sum() for r in runs]  # queued behind each call
    torch.cuda.synchronize()
    for r, a in zip(runs, after):
        _same(r, ref, "back to back")
        assert int(a.item()) == int(ref["placement"].to(torch.int32).sum().item())
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        o = _plan_outputs(L, E, M)
        with torch.cuda.graph(g, stream=s):
            B.ordermoe_plan(Wr, Xcal, L, E, d, N, kf, M, *TH, p, C, pi, o["sim"], o["counts"], o["group"],
                            o["n_groups"], o["theta"], o["importance"], o["placement"], o["used"],
                            o["status"], o["replicas"], o["cover"], o["covered"], ws)
    for v in o.values():
        v.fill_(7)
    g.replay()
    torch.cuda.synchronize()
    _same(o, ref, "graph replay")


def test_plan_argument_errors_and_nullable_coverage():
    """Argument errors come back before anything is enqueued; cover and
    covered may be omitted."""
    L, E, d, N, M, kf = 3, 64, 128, 700, 4, 6
    Wr, Xcal, p, C, pi = _plan_inputs(L, E, d, N, M, 9, False)
    ws = torch.empty(B.ordermoe_plan_workspace_bytes(L, E, N), dtype=torch.uint8, device=DEV)
    o = _plan_outputs(L, E, M)
    args = lambda **kw: dict(dict(sim=o["sim"], counts=o["counts"], group=o["group"], n_groups=o["n_groups"],
                                  theta=o["theta"], importance=o["importance"], placement=o["placement"],
                                  used=o["used"], status=o["status"], replicas=o["replicas"],
                                  cover=None, covered=None, workspace=ws), **kw)

    def call(L_=L, E_=E, M_=M, kf_=kf, **kw):
        a = args(**kw)
        B.ordermoe_plan(Wr, Xcal, L_, E_, d, N, kf_, M_, *TH, p, C, pi, a["sim"], a["counts"], a["group"],
                        a["n_groups"], a["theta"], a["importance"], a["placement"], a["used"], a["status"],
                        a["replicas"], a["cover"], a["covered"], a["workspace"])

    call()  # cover and covered omitted
    torch.cuda.synchronize()
    ref = _one_plan(Wr, Xcal, L, E, d, N, kf, M, p, C, pi, ws)
    torch.cuda.synchronize()
    for k in ("sim", "group", "placement", "used", "replicas"):
        assert torch.equal(o[k], ref[k]), k
    for kw, code in [(dict(importance=None), B.ERR_INVALID_ARG), (dict(workspace=ws[:1024]), B.ERR_INVALID_ARG),
                     (dict(M_=33), B.ERR_UNSUPPORTED_SHAPE), (dict(kf_=65), B.ERR_UNSUPPORTED_SHAPE),
                     (dict(E_=65), B.ERR_UNSUPPORTED_SHAPE)]:
        with pytest.raises(B.OrderMoEError) as ei:
            call(**kw)
        assert ei.value.code == code, kw
    torch.cuda.synchronize()


def test_plan_from_two_host_threads():
    """Two host threads, each on its own stream, call the plan at the same
    time with different inputs (the device's side stream and events are
    shared): every call writes its own single-call results."""
    import threading
    cases = [(13, 64, 128, 1500, 5, 6, 21), (9, 32, 128, 1200, 3, 4, 22)]
    prepared = []
    for L, E, d, N, M, kf, seed in cases:
        Wr, Xcal, p, C, pi = _plan_inputs(L, E, d, N, M, seed, True)
        ws = torch.empty(B.ordermoe_plan_workspace_bytes(L, E, N), dtype=torch.uint8, device=DEV)
        ref = _one_plan(Wr, Xcal, L, E, d, N, kf, M, p, C, pi, ws)
        prepared.append(((Wr, Xcal, L, E, d, N, kf, M, p, C, pi), ref))
    torch.cuda.synchronize()
    results = [[], []]
    errors = []

    def run(i):
        try:
            a, _ = prepared[i]
            s = torch.cuda.Stream()
            ws = torch.empty(B.ordermoe_plan_workspace_bytes(a[2], a[3], a[5]), dtype=torch.uint8,
                             device=DEV)
            with torch.cuda.stream(s):
                for _ in range(4):
                    results[i].append(_one_plan(*a, ws))
            s.synchronize()
        except Exception as e:  # reported below, in the test's thread
            errors.append(e)

    threads = [threading.Thread(target=run, args=(i,)) for i in range(2)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    torch.cuda.synchronize()
    assert not errors, errors
    for i in range(2):
        assert len(results[i]) == 4
        for r in results[i]:
            _same(r, prepared[i][1], "thread %d" % i)
