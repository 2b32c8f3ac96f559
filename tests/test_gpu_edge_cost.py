"""GPU parity of the edge cost of selection records (Eqs. 13-20), the
normalised utility (Eq. 23) and the weight adaptation (Eq. 45), against the
oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_17154_gb300 import binding as B
from paper_2607_17154_gb300 import synth
from tests.test_gpu_lookahead import stack_tables

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.lib()
    yield
    code, detail = B.ordermoe_device_error()
    assert code == 0, (code, detail)


def g(a, dt):
    return torch.as_tensor(np.ascontiguousarray(a)).to(device=DEV, dtype=dt)


def gpu_cost(target, chosen, server, home, buf, stride, E, sp):
    L, T, k = target.shape
    M = len(sp.F)
    d = torch.empty(T, dtype=torch.float64, device=DEV)
    q = torch.empty(T, dtype=torch.float64, device=DEV)
    n = torch.empty(T, dtype=torch.int32, device=DEV)
    B.ordermoe_trajectory_cost(g(target, torch.int32), g(chosen, torch.int32), g(server, torch.uint8),
                               g(home, torch.uint8), L, T, k, E, buf, stride, M,
                               g(sp.F, torch.float64), g(sp.B, torch.float64), g(sp.tau, torch.float64),
                               sp.z, sp.c, d, q, n)
    torch.cuda.synchronize()
    return d.cpu().numpy(), q.cpu().numpy(), n.cpu().numpy()


@pytest.mark.parametrize("L,T,k,E,M", [(1, 1, 1, 4, 2), (3, 1000, 2, 8, 4), (32, 128, 2, 8, 4),
                                       (5, 777, 6, 64, 8)])
def test_trajectory_cost_bit_exact_on_random_records(L, T, k, E, M):
    rng = np.random.default_rng(L * T + E)
    buf, stride, otabs = stack_tables(rng, L, E, M, 0.2, cheap_links=False)
    sp = synth.server_params(M, 4096, 14336, seed=0)
    sp.B = sp.B * rng.uniform(0.5, 2.0, (M, M))           # asymmetric links
    target = rng.integers(0, E, (L, T, k)).astype(np.int32)
    chosen = np.where(rng.random((L, T, k)) < 0.3, rng.integers(0, E, (L, T, k)), target).astype(np.int32)
    home = rng.integers(0, M, T).astype(np.uint8)
    server = np.where(rng.random((L, T, k)) < 0.5, home[None, :, None],
                      rng.integers(0, M, (L, T, k))).astype(np.uint8)
    got = gpu_cost(target, chosen, server, home, buf, stride, E, sp)
    Qtab = np.stack([t.Qtab for t in otabs])
    ref = oracle.trajectory_cost(target, chosen, server, home, sp.F, sp.B, sp.tau, sp.z, sp.c, Qtab)
    for name, a, b in zip(("delay", "loss", "moves"), got, ref):
        np.testing.assert_array_equal(a, b, err_msg=name)


def test_decode_trajectory_and_adaptation_follow_the_oracle():
    """32 Mixtral-shaped layers, batch 128: the GPU selects layer by layer
    (given logits), then prices the records; the delays, losses and transfers
    equal those of the oracle's own trajectory, and the utility and adapted
    weights follow."""
    w = synth.workload("decode_stack")
    L, T, E, k, M = w.L, w.T, w.E, w.k, w.M
    rng = np.random.default_rng(31)
    buf, stride, otabs = stack_tables(rng, L, E, M, w.qbar, cheap_links=True)
    sp = synth.server_params(M, 4096, 14336, seed=0)
    sp.tau[:] *= 1e-3
    logits = rng.standard_normal((L, T, E)).astype(np.float32)
    home = rng.integers(0, M, T).astype(np.uint8)
    gh = g(home, torch.uint8)
    gl, gq = gh.clone(), torch.zeros(T, device=DEV)
    rec = [torch.empty(L, T, k, dtype=dt, device=DEV) for dt in (torch.int32, torch.int32, torch.uint8)]
    for l in range(L):
        outs = [rec[0][l], torch.empty(T, k, device=DEV), rec[1][l], rec[2][l],
                torch.empty(T, k, dtype=torch.uint8, device=DEV)]
        B.ordermoe_route_select(None, None, g(logits[l], torch.float32), T, E, 0, k, 1,
                                buf[l * stride:(l + 1) * stride], gh, gl, gq, None, *outs)
    d = torch.empty(T, dtype=torch.float64, device=DEV)
    q = torch.empty(T, dtype=torch.float64, device=DEV)
    n = torch.empty(T, dtype=torch.int32, device=DEV)
    gF, gB, gt = g(sp.F, torch.float64), g(sp.B, torch.float64), g(sp.tau, torch.float64)
    B.ordermoe_trajectory_cost(rec[0], rec[1], rec[2], gh, L, T, k, E, buf, stride, M, gF, gB, gt,
                               sp.z, sp.c, d, q, n)
    # the oracle's own trajectory
    loc = home.copy(); qh = np.zeros(T, np.float32)
    o_t, o_c, o_s = [], [], []
    for l in range(L):
        idx, _ = oracle.topk(logits[l], k)
        ch, sv, _, loc, qh = oracle.select(idx, otabs[l], home, loc, qh)
        o_t.append(idx); o_c.append(ch); o_s.append(sv)
    Qtab = np.stack([t.Qtab for t in otabs])
    ref = oracle.trajectory_cost(np.stack(o_t), np.stack(o_c), np.stack(o_s), home, sp.F, sp.B,
                                 sp.tau, sp.z, sp.c, Qtab)
    np.testing.assert_array_equal(d.cpu().numpy(), ref[0])
    np.testing.assert_array_equal(q.cpu().numpy(), ref[1])
    np.testing.assert_array_equal(n.cpu().numpy(), ref[2])
    # utility and adaptation against a reference delay (bench.py takes it from
    # the exact-only records of the same deployment)
    out = torch.empty(5, dtype=torch.float64, device=DEV)
    dref = d * torch.as_tensor(rng.uniform(0.8, 1.0, T), dtype=torch.float64, device=DEV)
    B.ordermoe_utility(d, dref, q, T, w.qbar, 0.5, 0.5, 0.1, out)
    want = oracle.utility(ref[0], dref.cpu().numpy(), ref[1], w.qbar, 0.5, 0.5, 0.1)
    np.testing.assert_allclose(out.cpu().numpy(), want, rtol=1e-12, atol=0)


@pytest.mark.parametrize("T", [1, 100, 5000])
def test_utility_matches_oracle(T):
    rng = np.random.default_rng(T)
    d = rng.uniform(1e-3, 3e-2, T); r = d * rng.uniform(0.7, 1.3, T); q = rng.uniform(0, 0.05, T)
    out = torch.empty(5, dtype=torch.float64, device=DEV)
    B.ordermoe_utility(g(d, torch.float64), g(r, torch.float64), g(q, torch.float64), T, 0.1, 0.7, 0.3,
                       0.2, out)
    np.testing.assert_allclose(out.cpu().numpy(), oracle.utility(d, r, q, 0.1, 0.7, 0.3, 0.2),
                               rtol=1e-12, atol=1e-15)
    # the projection of Eq. 45 onto [0, 1]
    B.ordermoe_utility(g(d, torch.float64), g(d, torch.float64), g(0 * q, torch.float64), T, 0.1, 0.5,
                       0.5, 10.0, out)
    assert out[4].item() == 0.0 and out[3].item() == 1.0


def test_edge_cost_errors():
    E, M = 4, 2
    buf = torch.zeros(B.ordermoe_tables_bytes(E, M), dtype=torch.uint8, device=DEV)
    sp = synth.server_params(M, 256, 512, 0)
    bad = np.zeros((1, 3, 1), np.int32); bad[0, 1, 0] = E            # target out of range
    gpu_cost(bad, np.zeros((1, 3, 1), np.int32), np.zeros((1, 3, 1), np.uint8), np.zeros(3, np.uint8),
             buf, 0, E, sp)
    code, detail = B.ordermoe_device_error()
    assert code == B.DEV_BAD_INDEX and detail == 1
    out = torch.empty(5, dtype=torch.float64, device=DEV)
    one = torch.ones(4, dtype=torch.float64, device=DEV)
    ref = one.clone(); ref[2] = 0.0
    B.ordermoe_utility(one, ref, one, 4, 0.5, 0.5, 0.5, 0.1, out)
    code, detail = B.ordermoe_device_error()
    assert code == B.DEV_BAD_VALUE and detail == 2
    with pytest.raises(B.OrderMoEError) as ei:
        B.ordermoe_utility(one, one, one, 4, 0.0, 0.5, 0.5, 0.1, out)
    assert ei.value.code == B.ERR_INVALID_ARG
