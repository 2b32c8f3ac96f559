"""Parity of the remaining workload configurations at full size: the
fine-grained layer (E 64, top-6, Zipf homes) over the threshold sweep, and the
32-layer decode stack on the residual map, whose per-token trajectory state
(location and accumulated loss, Eqs. 36 and 44) is carried across layers."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_17154_gb300 import synth
from paper_2607_17154_gb300.layer import LayerStack, build_tables
from tests.helpers import assert_close_bf16
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
    layer = run_layer_check(w, seed=2, sample=512)
    kinds = layer.counters.cpu().numpy()
    assert kinds.sum() == w.T * w.k


def test_decode_stack_full_size_residual_teacher_forced():
    """One decode step of the 32-layer stack (batch 128, ~90 GB of expert
    weights resident) on the residual map h_{l+1} = h_l + y_l, each layer
    reading x_l = RMSNorm(h_l), with the selection state carried across the
    layers. The offline plan comes from the library's calibration pass along
    the same map; the oracle recomputes grouping and placement from its
    similarities and counts bit for bit. Teacher forcing per layer, every one
    of the 32 layers and all 128 tokens:
      * every integer decision (top-k, chosen expert and server, kind, location,
        accumulated loss, permutation) bit for bit from the GPU's own logits;
      * the router logits against the oracle's on the GPU's layer input;
      * the residual update against the oracle's combine of the GPU's expert
        outputs, and the next RMSNorm against the oracle's;
      * the expert outputs against the oracle's FFN at every fourth layer.
    Then the CUDA-graph replay of the whole step through the stack gives the
    per-layer chain's results bit for bit."""
    from paper_2607_17154_gb300 import binding as B
    from paper_2607_17154_gb300.layer import MoELayer, calibrate_stack
    from tests.helpers import check_layer_integers_full
    from tests.test_gpu_residual import _close_residual, assert_norm_close
    w = synth.workload("decode_stack")
    L, T, E, d, dff, k, M = w.L, w.T, w.E, w.d, w.dff, w.k, w.M
    seed = 11
    layers = []
    for l in range(L):
        inp = synth.layer_inputs(w, seed=seed, layer=l, device=DEV)
        layers.append({"W_r": inp["Wr"], "W1": inp["W1"], "W3": inp["W3"], "W2": inp["W2"]})
    home_np = synth.layer_inputs(w, seed=seed, with_ffn=False)["home"]
    home = torch.as_tensor(home_np).to(DEV)
    # offline plan along the residual map
    cal = calibrate_stack(layers, synth.calibration(w.n_cal, d, seed, device=DEV), k, M)
    group = torch.empty(L, E, dtype=torch.int32, device=DEV)
    ng = torch.empty(L, dtype=torch.int32, device=DEV)
    theta = torch.empty(L, dtype=torch.float32, device=DEV)
    x = torch.empty(L, M, E, dtype=torch.uint8, device=DEV)
    used = torch.empty(M, dtype=torch.float64, device=DEV)
    st = torch.empty(1, dtype=torch.int32, device=DEV)
    imp = torch.empty(L, E, dtype=torch.float64, device=DEV)
    B.ordermoe_place(cal["sim"], cal["counts"], L, E, M, w.theta_min, w.theta_max, w.theta, 0.5,
                     0.5, 0.5, 0.5, torch.ones(L, E, dtype=torch.float64, device=DEV),
                     torch.full((M,), L * E / M, dtype=torch.float64, device=DEV), group, ng, theta,
                     imp, x, used, st)
    torch.cuda.synchronize()
    assert st.item() == 0
    sims, counts = cal["sim"].cpu().numpy(), cal["counts"].cpu().numpy()
    thetas = [oracle.theta(l + 1, L, w.theta_min, w.theta_max, w.theta) for l in range(L)]
    np.testing.assert_array_equal(theta.cpu().numpy(), np.array(thetas, np.float32))
    o_groups, o_imps = [], []
    for l in range(L):
        g_, K_, _ = oracle.group(sims[l], counts[l], thetas[l])
        o_groups.append(g_); o_imps.append(oracle.importance(sims[l], counts[l], g_))
    np.testing.assert_array_equal(group.cpu().numpy(), np.stack(o_groups))
    o_x, _, rc = oracle.place(np.stack(o_groups), np.stack(o_imps), np.ones((L, E)),
                              np.full(M, L * E / M))
    assert rc == 0
    np.testing.assert_array_equal(x.cpu().numpy(), o_x)
    sp = synth.server_params(M, d, dff, seed)
    tabs = [build_tables(sims[l], o_groups[l], o_x[l], thetas[l], w.qbar, sp, DEV) for l in range(L)]
    o_tabs = [oracle.tables(sims[l], o_groups[l], o_x[l], thetas[l], w.qbar, sp.F, sp.B, sp.tau,
                            sp.z, sp.c, sp.omega_T, sp.omega_Q) for l in range(L)]
    del cal

    # the per-layer chain, checked layer by layer
    h0 = synth.hidden(T, d, seed + 5000, device=DEV)
    hs = [h0] + [torch.empty_like(h0) for _ in range(L)]
    xs = [torch.empty_like(h0) for _ in range(L + 1)]
    B.ordermoe_rmsnorm(hs[0], T, d, B.NORM_EPS, xs[0])
    loc, qhat = home.clone(), torch.zeros(T, device=DEV)
    torch.cuda.synchronize()
    assert_norm_close(synth.bits(xs[0]), oracle.rmsnorm(synth.bits(h0), B.NORM_EPS), "x_0")
    kinds = np.zeros(4, np.int64)
    for l in range(L):
        lay = layers[l]
        ml = MoELayer(lay["W_r"], lay["W1"], lay["W3"], lay["W2"], tabs[l], k, T)
        loc_in, q_in = loc.cpu().numpy(), qhat.cpu().numpy()
        ml.forward_residual(xs[l], hs[l], home, loc, qhat, hs[l + 1], xs[l + 1])
        torch.cuda.synchronize()
        xb, hb = synth.bits(xs[l]), synth.bits(hs[l])
        gpu = {"idx": ml.topk_idx.cpu().numpy(), "w": ml.topk_w.cpu().numpy(),
               "chosen": ml.chosen.cpu().numpy(), "server": ml.server.cpu().numpy(),
               "kind": ml.kind.cpu().numpy(), "loc": loc.cpu().numpy(), "qhat": qhat.cpu().numpy(),
               "offsets": ml.offsets.cpu().numpy(), "row_token": ml.row_token.cpu().numpy(),
               "row_of": ml.row_of.cpu().numpy(), "X_perm": synth.bits(ml.X_perm)}
        g_logits = ml.logits.cpu().numpy()
        Wrb = synth.bits(lay["W_r"])
        np.testing.assert_allclose(g_logits, oracle.router_logits(xb, Wrb), rtol=1e-3, atol=2e-3)
        idx, wt, chosen = check_layer_integers_full(g_logits, gpu, o_tabs[l], home_np, loc_in, q_in,
                                                    k, E, X_bits=xb, what="layer %d" % l)
        Yg = synth.bits(ml.Y_perm)[gpu["row_of"]]             # [T, k, d]
        ref_h = oracle.combine_residual(Yg.reshape(T * k, d),
                                        np.arange(T * k, dtype=np.int32).reshape(T, k), wt, hb)
        _close_residual(synth.bits(hs[l + 1]), ref_h, hb, wt, Yg, "h_%d" % (l + 1))
        assert_norm_close(synth.bits(xs[l + 1]), oracle.rmsnorm(synth.bits(hs[l + 1]), B.NORM_EPS),
                          "x_%d" % (l + 1))
        if l % 4 == 0:
            _, Yo = oracle.ffn_rows(np.repeat(xb, k, axis=0), chosen.reshape(-1),
                                    synth.bits(lay["W1"]), synth.bits(lay["W3"]),
                                    synth.bits(lay["W2"]))
            assert_close_bf16(Yg, Yo.reshape(T, k, d), what="expert outputs of layer %d" % l)
        kinds += np.bincount(gpu["kind"].ravel(), minlength=4)
        del ml
    # Property 2: the accumulated loss never exceeds the budget
    assert (qhat.cpu().numpy() <= np.float32(w.qbar)).all()
    assert kinds.sum() == L * T * k and kinds[1] + kinds[3] > 0    # substitutes happen
    chain = [loc.clone(), qhat.clone()] + [t.clone() for t in hs[1:] + xs[1:]]

    # the same step through the stack, captured as one CUDA graph and replayed
    stack = LayerStack(layers, tabs, k, T, DEV)
    hs2 = [h0] + [torch.zeros_like(h0) for _ in range(L)]
    xs2 = [torch.zeros_like(h0) for _ in range(L + 1)]
    loc2, q2 = home.clone(), torch.zeros(T, device=DEV)

    def reset():
        loc2.copy_(home)
        q2.zero_()

    graph = stack.capture_residual(hs2, xs2, home, loc2, q2, prologue=reset)
    for t in hs2[1:] + xs2[1:]:
        t.zero_()
    graph.replay()
    torch.cuda.synchronize()
    for a, b in zip(chain, [loc2, q2] + hs2[1:] + xs2[1:]):
        assert torch.equal(a, b)
