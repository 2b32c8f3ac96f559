"""GPU parity of the look-ahead selection (Eqs. 41-43): transition statistics
and the depth-H cost-to-go, against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_17154_gb300 import binding as B
from paper_2607_17154_gb300 import synth
from paper_2607_17154_gb300.layer import build_tables

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


@pytest.mark.parametrize("N,L,E,kf", [(5000, 4, 8, 2), (3000, 3, 64, 6), (100, 2, 5, 5)])
def test_transitions_given_logits_bit_exact(N, L, E, kf):
    rng = np.random.default_rng(N + E)
    logits = rng.standard_normal((N, L, E)).astype(np.float32)
    logits[:7] = 0.25                                   # ties
    cnt = torch.empty(L - 1, E, E, dtype=torch.int32, device=DEV)
    P = torch.empty(L - 1, E, E, dtype=torch.float32, device=DEV)
    B.ordermoe_transitions(torch.as_tensor(logits).to(DEV), N, L, E, kf, cnt, P)
    rc, rP = oracle.transitions(logits, kf)
    np.testing.assert_array_equal(cnt.cpu().numpy(), rc)
    np.testing.assert_array_equal(P.cpu().numpy(), rP)


def stack_tables(rng, L, E, M, qbar, cheap_links):
    """L layers' tables, random groups/placements, as one device buffer plus the
    oracle's own copies."""
    stride = B.ordermoe_tables_bytes(E, M)
    buf = torch.zeros(L * stride, dtype=torch.uint8, device=DEV)
    otabs = []
    for l in range(L):
        Wt = rng.standard_normal((E, 6)); Wt[:, 0] += 3.0 * (np.arange(E) % 3)
        nrm = np.linalg.norm(Wt, axis=1, keepdims=True)
        sim = ((Wt / nrm) @ (Wt / nrm).T).astype(np.float32); np.fill_diagonal(sim, 1.0)
        group = (np.arange(E) % 3).astype(np.int32)
        x = (rng.random((M, E)) < 0.35).astype(np.uint8)
        for e in range(E):
            if not x[:, e].any():
                x[rng.integers(M), e] = 1
        sp = synth.server_params(M, 4096, 14336, seed=l)
        if cheap_links:
            sp.tau[:] *= 1e-3
        theta = 0.2
        build_tables(sim, group, x, theta, qbar, sp, DEV, out=buf[l * stride:(l + 1) * stride])
        otabs.append(oracle.tables(sim, group, x, theta, qbar, sp.F, sp.B, sp.tau, sp.z, sp.c,
                                   sp.omega_T, sp.omega_Q))
    return buf, stride, otabs


@pytest.mark.parametrize("E,M,k,H,cheap", [(8, 4, 2, 1, True), (8, 4, 2, 2, True), (8, 4, 2, 3, True),
                                           (16, 4, 3, 3, False), (6, 3, 2, 4, True), (32, 8, 2, 2, True),
                                           # H = 3 with 8 servers and dear links: about half the
                                           # tokens have more than 512 pairs in their first slot
                                           # whose Phi^(1) is not tabulated (up to about 1100), more
                                           # than the kernel lists (the rest evaluated in place);
                                           # with 4 servers at most about 215
                                           (16, 8, 3, 3, False),
                                           # H = 4: the Phi^(2) table used (cheap substitutes) and
                                           # bypassed when budget checks can fail (dear ones)
                                           (8, 4, 2, 4, False), (16, 4, 3, 4, True), (12, 5, 2, 4, False)])
def test_route_select_lookahead_given_logits_bit_exact(E, M, k, H, cheap):
    rng = np.random.default_rng(E * 10 + H)
    T = 300
    qbar = 0.2
    buf, stride, otabs = stack_tables(rng, H, E, M, qbar, cheap)
    P = rng.random((max(H - 1, 1), E, E)).astype(np.float32)
    P[P < 0.5] = 0
    P = (P / np.maximum(P.sum(axis=2, keepdims=True), 1e-9)).astype(np.float32)
    logits = rng.standard_normal((T, E)).astype(np.float32)
    home = rng.integers(0, M, T).astype(np.uint8)
    loc = np.where(rng.random(T) < 0.5, home, rng.integers(0, M, T)).astype(np.uint8)
    qhat = (rng.random(T) * 0.1).astype(np.float32)
    g = [torch.empty(T, k, dtype=dt, device=DEV)
         for dt in (torch.int32, torch.float32, torch.int32, torch.uint8, torch.uint8)]
    gl = torch.as_tensor(loc).to(DEV); gq = torch.as_tensor(qhat).to(DEV)
    B.ordermoe_route_select_lookahead(None, None, torch.as_tensor(logits).to(DEV), T, E, 0, k, 1, buf,
                                      stride, H, torch.as_tensor(P).to(DEV) if H > 1 else None,
                                      torch.as_tensor(home).to(DEV), gl, gq, None, *g)
    idx, _ = oracle.topk(logits, k)
    ref = oracle.select_lookahead(idx, otabs[:H], P[:H - 1], home, loc, qhat)
    for name, got, want in zip(("chosen", "server", "kind"), (g[2], g[3], g[4]), ref[:3]):
        np.testing.assert_array_equal(got.cpu().numpy(), want, err_msg=name)
    np.testing.assert_array_equal(gl.cpu().numpy(), ref[3])
    np.testing.assert_array_equal(gq.cpu().numpy(), ref[4])
    if H > 1:
        myo = oracle.select(idx, otabs[0], home, loc, qhat)
        print("decisions changed by the look-ahead:", int((myo[0] != ref[0]).sum() + (myo[1] != ref[1]).sum()))


def test_lookahead_horizon_one_equals_route_select():
    rng = np.random.default_rng(5)
    E, M, k, T = 8, 4, 2, 200
    buf, stride, otabs = stack_tables(rng, 1, E, M, 0.2, True)
    logits = torch.as_tensor(rng.standard_normal((T, E)).astype(np.float32)).to(DEV)
    home = torch.as_tensor(rng.integers(0, M, T).astype(np.uint8)).to(DEV)
    outs = []
    for fn in ("plain", "lookahead"):
        g = [torch.empty(T, k, dtype=dt, device=DEV)
             for dt in (torch.int32, torch.float32, torch.int32, torch.uint8, torch.uint8)]
        if fn == "plain":
            B.ordermoe_route_select(None, None, logits, T, E, 0, k, 1, buf, home, None, None, None, *g)
        else:
            B.ordermoe_route_select_lookahead(None, None, logits, T, E, 0, k, 1, buf, stride, 1, None,
                                              home, None, None, None, *g)
        outs.append([t.cpu() for t in g])
    for a, b in zip(*outs):
        assert torch.equal(a, b)


def test_decode_stack_with_lookahead_h3_follows_the_oracle():
    """32 Mixtral-shaped routers, batch 128, H = 3: each layer looks two layers
    ahead with the transition statistics of the calibration logits. The
    oracle follows every token through the 32 selections (fed the same fp32
    logits, so each decision is compared exactly)."""
    w = synth.workload("decode_stack")
    L, T, E, k, M = w.L, w.T, w.E, w.k, w.M
    H = 3
    rng = np.random.default_rng(21)
    buf, stride, otabs = stack_tables(rng, L, E, M, w.qbar, cheap_links=True)
    cal = rng.standard_normal((4096, L, E)).astype(np.float32)
    _, P = oracle.transitions(cal, k)
    gP = torch.as_tensor(P).to(DEV)
    logits = rng.standard_normal((L, T, E)).astype(np.float32)
    home = rng.integers(0, M, T).astype(np.uint8)
    gl = torch.as_tensor(home).to(DEV); gq = torch.zeros(T, device=DEV)
    gh = torch.as_tensor(home).to(DEV)
    gch = []
    for l in range(L):
        Hl = min(H, L - l)
        g = [torch.empty(T, k, dtype=dt, device=DEV)
             for dt in (torch.int32, torch.float32, torch.int32, torch.uint8, torch.uint8)]
        B.ordermoe_route_select_lookahead(None, None, torch.as_tensor(logits[l]).to(DEV), T, E, 0, k, 1,
                                          buf[l * stride:], stride, Hl,
                                          gP[l:l + Hl - 1].contiguous() if Hl > 1 else None,
                                          gh, gl, gq, None, *g)
        gch.append(g[2].cpu().numpy())
    loc = home.copy(); q = np.zeros(T, np.float32)
    for l in range(L):
        Hl = min(H, L - l)
        idx, _ = oracle.topk(logits[l], k)
        ch, sv, kd, loc, q = oracle.select_lookahead(idx, otabs[l:l + Hl], P[l:l + Hl - 1], home, loc, q)
        np.testing.assert_array_equal(gch[l], ch, err_msg="layer %d" % l)
    np.testing.assert_array_equal(gl.cpu().numpy(), loc)
    np.testing.assert_array_equal(gq.cpu().numpy(), q)
    assert (q <= np.float32(w.qbar)).all()


@pytest.mark.parametrize("E,M,k,H", [(8, 4, 2, 3), (16, 6, 4, 2), (64, 8, 6, 2)])
def test_router_path_lookahead_bit_exact(E, M, k, H):
    """Router GEMM on the tensor cores, then the warp-per-token look-ahead
    pass: the decisions follow the oracle given the logits the router wrote
    (T spans three 128-row router tiles with a ragged tail)."""
    rng = np.random.default_rng(E + 100 * H)
    T, d = 300, 256
    buf, stride, otabs = stack_tables(rng, H, E, M, 0.25, cheap_links=True)
    P = rng.random((H - 1, E, E)).astype(np.float32)
    P[P < 0.6] = 0
    P = (P / np.maximum(P.sum(axis=2, keepdims=True), 1e-9)).astype(np.float32)
    X = torch.randn(T, d, device=DEV).to(torch.bfloat16)
    W_r = (torch.randn(E, d, device=DEV) * 0.2).to(torch.bfloat16)
    home = rng.integers(0, M, T).astype(np.uint8)
    loc = np.where(rng.random(T) < 0.5, home, rng.integers(0, M, T)).astype(np.uint8)
    qhat = (rng.random(T) * 0.1).astype(np.float32)
    g = [torch.empty(T, k, dtype=dt, device=DEV)
         for dt in (torch.int32, torch.float32, torch.int32, torch.uint8, torch.uint8)]
    lg = torch.empty(T, E, device=DEV)
    cnt = torch.zeros(4, dtype=torch.int32, device=DEV)
    gl = torch.as_tensor(loc).to(DEV); gq = torch.as_tensor(qhat).to(DEV)
    B.ordermoe_route_select_lookahead(X, W_r, None, T, E, d, k, 1, buf, stride, H,
                                      torch.as_tensor(P).to(DEV), torch.as_tensor(home).to(DEV),
                                      gl, gq, lg, *g, counters=cnt)
    logits = lg.cpu().numpy()
    idx, _ = oracle.topk(logits, k)
    np.testing.assert_array_equal(g[0].cpu().numpy(), idx)
    ch, sv, kd, rl, rq = oracle.select_lookahead(idx, otabs, P, home, loc, qhat)
    np.testing.assert_array_equal(g[2].cpu().numpy(), ch)
    np.testing.assert_array_equal(g[3].cpu().numpy(), sv)
    np.testing.assert_array_equal(g[4].cpu().numpy(), kd)
    np.testing.assert_array_equal(gl.cpu().numpy(), rl)
    np.testing.assert_array_equal(gq.cpu().numpy(), rq)
    np.testing.assert_array_equal(cnt.cpu().numpy(), np.bincount(kd.ravel(), minlength=4))


def test_lookahead_skips_a_nan_token_and_reports_it():
    rng = np.random.default_rng(9)
    E, M, k, T, H = 8, 4, 2, 70, 2
    buf, stride, otabs = stack_tables(rng, H, E, M, 0.2, cheap_links=True)
    P = np.full((1, E, E), 1.0 / E, np.float32)
    logits = rng.standard_normal((T, E)).astype(np.float32)
    bad = logits.copy(); bad[3, 5] = np.nan
    home = rng.integers(0, M, T).astype(np.uint8)
    g = [torch.empty(T, k, dtype=dt, device=DEV)
         for dt in (torch.int32, torch.float32, torch.int32, torch.uint8, torch.uint8)]
    gl = torch.as_tensor(home).to(DEV); gq = torch.zeros(T, device=DEV)
    B.ordermoe_route_select_lookahead(None, None, torch.as_tensor(bad).to(DEV), T, E, 0, k, 1, buf,
                                      stride, H, torch.as_tensor(P).to(DEV),
                                      torch.as_tensor(home).to(DEV), gl, gq, None, *g)
    code, detail = B.ordermoe_device_error()
    assert code == B.DEV_NAN_LOGIT and detail == 3
    idx, _ = oracle.topk(logits, k)
    ch, sv, kd, rl, rq = oracle.select_lookahead(idx, otabs, P, home, home.copy(),
                                                 np.zeros(T, np.float32))
    keep = np.arange(T) != 3
    np.testing.assert_array_equal(g[2].cpu().numpy()[keep], ch[keep])
    np.testing.assert_array_equal(g[3].cpu().numpy()[keep], sv[keep])
    np.testing.assert_array_equal(gl.cpu().numpy()[keep], rl[keep])
    assert gl[3].item() == home[3] and gq[3].item() == 0.0       # state of the NaN token kept
    assert (g[0][3] == -1).all().item()


def test_layer_stack_lookahead_through_layer_forward():
    """Six small layers through ordermoe_layer_forward with H = 3 (router on the
    tensor cores, tables of all layers in one stack, transition matrices
    between them): the carried location and loss follow the oracle's
    look-ahead selection on the oracle's own router logits, for every token
    whose top-k has no near tie at any layer."""
    from paper_2607_17154_gb300.layer import LayerStack
    rng = np.random.default_rng(44)
    L, T, E, k, M, d, dff, H = 6, 300, 8, 2, 4, 256, 512, 3
    buf, stride, otabs = stack_tables(rng, L, E, M, 0.3, cheap_links=True)
    P = rng.random((L - 1, E, E)).astype(np.float32)
    P[P < 0.5] = 0
    P = (P / np.maximum(P.sum(axis=2, keepdims=True), 1e-9)).astype(np.float32)
    layers, Wrb = [], []
    for l in range(L):
        Wr = synth.router_weights(E, d, 2, seed=70 + l, device=DEV)
        W1, W3, W2 = synth.ffn_weights(E, d, dff, seed=80 + l, device=DEV)
        layers.append({"W_r": Wr, "W1": W1, "W3": W3, "W2": W2})
        Wrb.append(synth.bits(Wr))
    stack = LayerStack(layers, buf, k, T, DEV, H=H, stride=stride, P=torch.as_tensor(P).to(DEV))
    Xs = [synth.hidden(T, d, 90 + l, device=DEV) for l in range(L)]
    ys = [torch.empty(T, d, dtype=torch.bfloat16, device=DEV) for _ in range(L)]
    home_np = rng.integers(0, M, T).astype(np.uint8)
    home = torch.as_tensor(home_np).to(DEV)
    loc, qhat = home.clone(), torch.zeros(T, device=DEV)
    counters = torch.zeros(4, dtype=torch.int32, device=DEV)
    stack.step(Xs, home, loc, qhat, ys, counters)
    torch.cuda.synchronize()
    assert counters.sum().item() == L * T * k
    o_loc, o_q = home_np.copy(), np.zeros(T, np.float32)
    clear = np.ones(T, bool)
    for l in range(L):
        logits = oracle.router_logits(synth.bits(Xs[l]), Wrb[l])
        srt = -np.sort(-logits.astype(np.float64), axis=1)
        clear &= np.abs(np.diff(srt[:, :k + 1], axis=1)).min(axis=1) > 1e-3
        idx, _ = oracle.topk(logits, k)
        Hl = min(H, L - l)
        _, _, _, o_loc, o_q = oracle.select_lookahead(idx, otabs[l:l + Hl], P[l:l + Hl - 1], home_np,
                                                      o_loc, o_q)
    assert clear.mean() > 0.6
    np.testing.assert_array_equal(loc.cpu().numpy()[clear], o_loc[clear])
    np.testing.assert_array_equal(qhat.cpu().numpy()[clear], o_q[clear])
    assert torch.isfinite(ys[-1].float()).all()


def test_layer_stack_graph_replay_equals_eager_step():
    """A step captured as one CUDA graph and replayed gives the eager step's
    outputs bit for bit (location, loss, every layer's y), with look-ahead."""
    from paper_2607_17154_gb300.layer import LayerStack
    rng = np.random.default_rng(45)
    L, T, E, k, M, d, dff, H = 4, 128, 8, 2, 4, 256, 512, 3
    buf, stride, _ = stack_tables(rng, L, E, M, 0.3, cheap_links=True)
    P = rng.random((L - 1, E, E)).astype(np.float32)
    P = (P / P.sum(axis=2, keepdims=True)).astype(np.float32)
    layers = []
    for l in range(L):
        W1, W3, W2 = synth.ffn_weights(E, d, dff, seed=180 + l, device=DEV)
        layers.append({"W_r": synth.router_weights(E, d, 2, seed=170 + l, device=DEV),
                       "W1": W1, "W3": W3, "W2": W2})
    stack = LayerStack(layers, buf, k, T, DEV, H=H, stride=stride, P=torch.as_tensor(P).to(DEV))
    Xs = [synth.hidden(T, d, 190 + l, device=DEV) for l in range(L)]
    home = torch.as_tensor(rng.integers(0, M, T).astype(np.uint8)).to(DEV)
    outs = []
    for mode in ("eager", "graph"):
        ys = [torch.zeros(T, d, dtype=torch.bfloat16, device=DEV) for _ in range(L)]
        loc, qhat = home.clone(), torch.zeros(T, device=DEV)

        def reset():
            loc.copy_(home)
            qhat.zero_()
        if mode == "eager":
            reset()
            stack.step(Xs, home, loc, qhat, ys)
        else:
            g = stack.capture(Xs, home, loc, qhat, ys, prologue=reset)
            for y in ys:
                y.zero_()
            loc.fill_(0)
            g.replay()
        torch.cuda.synchronize()
        outs.append([loc.clone(), qhat.clone()] + [y.clone() for y in ys])
    for a, b in zip(*outs):
        assert torch.equal(a, b)


def test_residual_stack_lookahead_teacher_forced():
    """Six small layers on the residual map (each layer reads RMSNorm of the
    residual stream) through ordermoe_layer_forward_residual with H = 3: with
    the oracle fed each layer's recorded router logits (teacher forcing), the
    look-ahead selection carries the same location and accumulated loss for
    every token, bit for bit, near ties included; the recorded logits match
    the oracle's on the GPU's layer inputs; a CUDA-graph replay of the step
    gives the eager step's results bit for bit."""
    from paper_2607_17154_gb300.layer import LayerStack
    rng = np.random.default_rng(46)
    L, T, E, k, M, d, dff, H = 6, 300, 8, 2, 4, 256, 512, 3
    buf, stride, otabs = stack_tables(rng, L, E, M, 0.3, cheap_links=True)
    P = rng.random((L - 1, E, E)).astype(np.float32)
    P[P < 0.5] = 0
    P = (P / np.maximum(P.sum(axis=2, keepdims=True), 1e-9)).astype(np.float32)
    layers, Wrb = [], []
    for l in range(L):
        Wr = synth.router_weights(E, d, 2, seed=270 + l, device=DEV)
        W1, W3, W2 = synth.ffn_weights(E, d, dff, seed=280 + l, device=DEV)
        layers.append({"W_r": Wr, "W1": W1, "W3": W3, "W2": W2})
        Wrb.append(synth.bits(Wr))
    stack = LayerStack(layers, buf, k, T, DEV, H=H, stride=stride, P=torch.as_tensor(P).to(DEV))
    home_np = rng.integers(0, M, T).astype(np.uint8)
    home = torch.as_tensor(home_np).to(DEV)
    h0 = synth.hidden(T, d, 290, device=DEV)
    outs = []
    for mode in ("eager", "graph"):
        hs = [h0] + [torch.zeros_like(h0) for _ in range(L)]
        xs = [torch.zeros_like(h0) for _ in range(L + 1)]
        loc, qhat = home.clone(), torch.zeros(T, device=DEV)
        logits = torch.zeros(L, T, E, device=DEV)

        def reset():
            loc.copy_(home)
            qhat.zero_()
        if mode == "eager":
            counters = torch.zeros(4, dtype=torch.int32, device=DEV)
            reset()
            stack.step_residual(hs, xs, home, loc, qhat, counters=counters, logits=logits)
            torch.cuda.synchronize()
            assert counters.sum().item() == L * T * k
            lg = logits.cpu().numpy()
            o_loc, o_q = home_np.copy(), np.zeros(T, np.float32)
            for l in range(L):
                np.testing.assert_allclose(lg[l], oracle.router_logits(synth.bits(xs[l]), Wrb[l]),
                                           rtol=1e-3, atol=2e-3)
                idx, _ = oracle.topk(lg[l], k)
                Hl = min(H, L - l)
                _, _, _, o_loc, o_q = oracle.select_lookahead(idx, otabs[l:l + Hl], P[l:l + Hl - 1],
                                                              home_np, o_loc, o_q)
            np.testing.assert_array_equal(loc.cpu().numpy(), o_loc)
            np.testing.assert_array_equal(qhat.cpu().numpy().view(np.uint32), o_q.view(np.uint32))
            assert torch.isfinite(hs[-1].float()).all()
        else:
            g = stack.capture_residual(hs, xs, home, loc, qhat, prologue=reset)
            for t in hs[1:] + xs:
                t.zero_()
            loc.fill_(0)
            g.replay()
            torch.cuda.synchronize()
        outs.append([loc.clone(), qhat.clone()] + [t.clone() for t in hs[1:] + xs])
    for a, b in zip(*outs):
        assert torch.equal(a, b)
