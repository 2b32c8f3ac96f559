"""Parity of the remaining workload configurations at full size: the
fine-grained layer (E 64, top-6, Zipf homes) over the threshold sweep, and the
32-layer decode stack whose per-token trajectory state (location and
accumulated loss, Eqs. 36 and 44) is carried across layers."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_17154_gb300 import synth
from paper_2607_17154_gb300.layer import LayerStack, build_tables
from tests.helpers import (assert_close_bf16, assert_close_combined, bits_to_f,
                           oracle_layer_tokens)
from tests.test_gpu_path import run_layer_check

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2607_17154_gb300 import binding as B
    B.lib()
    yield
    code, detail = B.ordermoe_device_error()
    assert code == 0, (code, detail)


@pytest.mark.parametrize("theta", [0.3, 0.5, 0.7])
def test_fine_grained_full_size_threshold_sweep(theta):
    w = synth.workload("fine_grained", theta=theta)
    layer = run_layer_check(w, seed=2, sample=48)
    kinds = layer.counters.cpu().numpy()
    assert kinds.sum() == w.T * w.k


def oracle_stack_plan(Wr_layers_bits, Xcal_bits, w):
    """Oracle plan of all layers: Eqs. 3-6 per layer, then placement with the
    used memory carried across layers (Alg. 1)."""
    L = len(Wr_layers_bits)
    sims, groups, imps, thetas = [], [], [], []
    for l, Wb in enumerate(Wr_layers_bits):
        sim, H = oracle.similarity(Wb, Xcal_bits, return_H=True)
        counts = oracle.expert_counts(np.ascontiguousarray(H.T), w.k)
        th = oracle.theta(l + 1, L, w.theta_min, w.theta_max, w.theta)
        g, K, _ = oracle.group(sim, counts, th)
        sims.append(sim); groups.append(g); thetas.append(th)
        imps.append(oracle.importance(sim, counts, g))
    x, used, rc = oracle.place(np.stack(groups), np.stack(imps), np.ones((L, w.E)),
                               np.full(w.M, L * w.E / w.M))
    assert rc == 0
    return sims, groups, thetas, x


def test_decode_stack_full_size_sampled():
    """One decode step of the 32-layer stack (batch 128, ~90 GB of expert
    weights resident). Each layer's input is a fresh seeded N(0,1) draw (the
    hidden state entering that MoE layer); the selection state is carried. The
    oracle follows each sampled token through all 32 selections and recomputes
    the expert FFN and combine at three sampled layers."""
    w = synth.workload("decode_stack")
    L, T, E, d, dff, k = w.L, w.T, w.E, w.d, w.dff, w.k
    seed = 11
    layers = [synth.layer_inputs(w, seed=seed, layer=l, device=DEV) for l in range(L)]
    Xcal = synth.calibration(w.n_cal, d, seed)
    sims, groups, thetas, x = oracle_stack_plan([synth.bits(l["Wr"]) for l in layers],
                                                synth.bits(Xcal), w)
    sp = synth.server_params(w.M, d, dff, seed)
    tabs = [build_tables(sims[l], groups[l], x[l], thetas[l], w.qbar, sp, DEV) for l in range(L)]
    stack = LayerStack([{"W_r": l["Wr"], "W1": l["W1"], "W3": l["W3"], "W2": l["W2"]} for l in layers],
                       tabs, k, T, DEV)
    Xs = [synth.hidden(T, d, seed + 5000 + l, device=DEV) for l in range(L)]
    ys = [torch.empty(T, d, dtype=torch.bfloat16, device=DEV) for _ in range(L)]
    home_np = layers[0]["home"]
    home = torch.as_tensor(home_np).to(DEV)
    loc = home.clone()
    qhat = torch.zeros(T, device=DEV)
    counters = torch.zeros(4, dtype=torch.int32, device=DEV)
    stack.step(Xs, home, loc, qhat, ys, counters)
    torch.cuda.synchronize()
    assert counters.sum().item() == L * T * k

    o_tabs = [oracle.tables(sims[l], groups[l], x[l], thetas[l], w.qbar, sp.F, sp.B, sp.tau,
                            sp.z, sp.c, sp.omega_T, sp.omega_Q) for l in range(L)]
    toks = np.sort(np.random.default_rng(seed).choice(T, 24, replace=False))
    check_layers = (0, L // 2, L - 1)
    o_loc = home_np[toks].copy()
    o_q = np.zeros(len(toks), np.float32)
    clear = np.ones(len(toks), bool)
    Xbits = [synth.bits(X)[toks] for X in Xs]
    for l in range(L):
        Wrb = synth.bits(layers[l]["Wr"])
        if l in check_layers:
            ref = oracle_layer_tokens(np.arange(len(toks)), Xbits[l], Wrb, synth.bits(layers[l]["W1"]),
                                      synth.bits(layers[l]["W3"]), synth.bits(layers[l]["W2"]),
                                      o_tabs[l], home_np[toks], o_loc, o_q, k)
            clear &= ref["margin"] > 1e-4
            c = clear
            assert_close_combined(synth.bits(ys[l])[toks][c], ref["y"][c], ref["w"][c], ref["Y"][c],
                                  what="y of layer %d" % l)
            o_loc, o_q = ref["loc"], ref["qhat"]
        else:
            logits = oracle.router_logits(Xbits[l], Wrb)
            srt = -np.sort(-logits.astype(np.float64), axis=1)
            clear &= np.abs(np.diff(srt[:, :k + 1], axis=1)).min(axis=1) > 1e-4
            idx, _ = oracle.topk(logits, k)
            _, _, _, o_loc, o_q = oracle.select(idx, o_tabs[l], home_np[toks], o_loc, o_q)
    assert clear.mean() > 0.5
    np.testing.assert_array_equal(loc.cpu().numpy()[toks][clear], o_loc[clear])
    np.testing.assert_array_equal(qhat.cpu().numpy()[toks][clear], o_q[clear])
    # Property 2: the accumulated loss never exceeds the budget
    assert (qhat.cpu().numpy() <= np.float32(w.qbar)).all()
