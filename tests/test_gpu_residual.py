"""GPU parity of the residual map between stacked layers (RMSNorm, the
residual combine) and of the transition statistics over strided logits,
through the C ABI, against the CPU oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_17154_gb300 import binding as B
from paper_2607_17154_gb300 import synth
from tests.helpers import bits_to_f

pytestmark = pytest.mark.gpu

DEV = "cuda:0"
EPS = B.NORM_EPS


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.lib()
    yield
    code, detail = B.ordermoe_device_error()
    assert code == 0, (code, detail)


def bf(bits):
    return synth.from_bits(bits).to(DEV)


def assert_norm_close(got_bits, ref_bits, what):
    """RMSNorm outputs: both sides round h / rms once to bf16 from values that
    agree to ~1e-6 relative (fp32 sum of squares and correctly rounded
    rsqrt against fp64), so they differ by at most one bf16 step, and rarely."""
    g = bits_to_f(got_bits).astype(np.float64)
    r = bits_to_f(ref_bits).astype(np.float64)
    bad = np.abs(g - r) > 2.0 ** -7 * np.abs(r) + 1e-30
    assert not bad.any(), "%s: %d elements differ by more than one bf16 step" % (what, bad.sum())
    assert (got_bits == ref_bits).mean() > 0.99, what


@pytest.mark.parametrize("T,d,scale", [(37, 4096, 1.0), (1000, 2048, 7.5), (1, 8, 0.01),
                                       (129, 264, 300.0)])
def test_rmsnorm_matches_oracle(T, d, scale):
    rng = np.random.default_rng(T + d)
    hb = synth.bits(torch.as_tensor(rng.standard_normal((T, d)) * scale, dtype=torch.float32)
                    .to(torch.bfloat16))
    x = torch.empty(T, d, dtype=torch.bfloat16, device=DEV)
    B.ordermoe_rmsnorm(bf(hb), T, d, EPS, x)
    torch.cuda.synchronize()
    assert_norm_close(synth.bits(x), oracle.rmsnorm(hb, EPS), "x")


@pytest.mark.parametrize("T,k,d", [(128, 2, 4096), (333, 6, 2048), (5, 8, 8), (64, 1, 256)])
def test_combine_residual_norm_matches_oracle(T, k, d):
    """h_out = h + sum_j w_j Y_j against the oracle's fp64 sum (fp32 FMAs in
    slot order on the GPU: within 2e-2 of the magnitude the sum carries,
    |h| + sum_j |w_j| |Y_j|, plus 1e-2), and x_out = RMSNorm(h_out) against
    the oracle's RMSNorm of the GPU's own h_out."""
    rng = np.random.default_rng(7 * T + k)
    R = T * k
    Yb = synth.bits(torch.as_tensor(rng.standard_normal((R, d)) * 2, dtype=torch.float32)
                    .to(torch.bfloat16))
    hb = synth.bits(torch.as_tensor(rng.standard_normal((T, d)) * 3, dtype=torch.float32)
                    .to(torch.bfloat16))
    row_of = rng.permutation(R).astype(np.int32).reshape(T, k)
    w = rng.random((T, k)).astype(np.float32)
    w /= w.sum(axis=1, keepdims=True)
    h_out = torch.full((T, d), float("nan"), dtype=torch.bfloat16, device=DEV)
    x_out = torch.full((T, d), float("nan"), dtype=torch.bfloat16, device=DEV)
    B.ordermoe_combine_residual_norm(bf(Yb), torch.as_tensor(row_of).to(DEV),
                                     torch.as_tensor(w).to(DEV), bf(hb), T, k, d, EPS, h_out, x_out)
    torch.cuda.synchronize()
    ref = bits_to_f(oracle.combine_residual(Yb, row_of, w, hb)).astype(np.float64)
    got = bits_to_f(synth.bits(h_out)).astype(np.float64)
    scale = np.abs(bits_to_f(hb)) + np.einsum("tk,tkd->td", w.astype(np.float64),
                                              np.abs(bits_to_f(Yb)[row_of]).astype(np.float64))
    assert (np.abs(got - ref) <= 1e-2 + 2e-2 * scale).all()
    assert_norm_close(synth.bits(x_out), oracle.rmsnorm(synth.bits(h_out), EPS), "x_out")


def test_combine_residual_norm_argument_errors_and_bad_rows():
    T, k, d = 4, 2, 64
    z = lambda *s: torch.zeros(*s, dtype=torch.bfloat16, device=DEV)
    Y, h, ho, xo = z(T * k, d), z(T, d), z(T, d), z(T, d)
    rof = torch.arange(T * k, dtype=torch.int32, device=DEV).view(T, k)
    w = torch.full((T, k), 0.5, device=DEV)
    with pytest.raises(B.OrderMoEError) as ei:
        B.ordermoe_combine_residual_norm(Y, rof, w, h, T, k, d, EPS, h, xo)   # h_out is h
    assert ei.value.code == B.ERR_INVALID_ARG
    with pytest.raises(B.OrderMoEError) as ei:
        B.ordermoe_combine_residual_norm(Y, rof, w, h, T, k, d, 0.0, ho, xo)  # eps must be > 0
    assert ei.value.code == B.ERR_INVALID_ARG
    with pytest.raises(B.OrderMoEError) as ei:
        B.ordermoe_rmsnorm(h, T, 12, EPS, xo)                                  # d % 8 != 0
    assert ei.value.code == B.ERR_UNSUPPORTED_SHAPE
    # a row index outside Y_perm is reported, and that token is left untouched
    bad = rof.clone(); bad[2, 1] = T * k
    ho.fill_(7.0); xo.fill_(7.0)
    B.ordermoe_combine_residual_norm(Y, bad, w, h + 1, T, k, d, EPS, ho, xo)
    torch.cuda.synchronize()
    code, detail = B.ordermoe_device_error()
    assert code == B.DEV_BAD_INDEX and detail == 2
    assert (ho[2] == 7.0).all() and (xo[2] == 7.0).all()
    assert (ho[0] == 1.0).all() and (xo[0] == 1.0).all()


@pytest.mark.parametrize("N,L,E,kf", [(5000, 4, 8, 2), (777, 3, 64, 6), (1, 2, 5, 5)])
def test_transitions_strided_layer_major_matches_oracle(N, L, E, kf):
    """Eq. 41 over layer-major logits [L][N][E] (as a stack's calibration pass
    records them): bit for bit the oracle's counts and P on the same logits,
    and the token-major entry point on the transposed copy."""
    rng = np.random.default_rng(N + L + E)
    lm = rng.standard_normal((L, N, E)).astype(np.float32)
    lm[:, ::7, 1] = lm[:, ::7, 0]          # exact ties straddling the top-k boundary
    tm = np.ascontiguousarray(lm.transpose(1, 0, 2))
    ref_c, ref_P = oracle.transitions(tm, kf)
    outs = []
    for strided in (True, False):
        c = torch.empty(L - 1, E, E, dtype=torch.int32, device=DEV)
        P = torch.empty(L - 1, E, E, dtype=torch.float32, device=DEV)
        if strided:
            B.ordermoe_transitions_strided(torch.as_tensor(lm).to(DEV), N, L, E, kf, E, N * E, c, P)
        else:
            B.ordermoe_transitions(torch.as_tensor(tm).to(DEV), N, L, E, kf, c, P)
        torch.cuda.synchronize()
        outs.append((c.cpu().numpy(), P.cpu().numpy()))
    for c, P in outs:
        np.testing.assert_array_equal(c, ref_c.reshape(c.shape))
        np.testing.assert_array_equal(P.view(np.uint32), ref_P.reshape(P.shape).view(np.uint32))


def _close_residual(got_bits, ref_bits, h_bits, w, Y_bits, what):
    """h + sum_j w_j Y_j: within 1e-2 + 2e-2 (|h| + sum_j |w_j| |Y_j|)."""
    g = bits_to_f(got_bits).astype(np.float64)
    r = bits_to_f(ref_bits).astype(np.float64)
    scale = np.abs(bits_to_f(h_bits)) + np.einsum("tk,tkd->td", np.abs(w).astype(np.float64),
                                                  np.abs(bits_to_f(Y_bits)).astype(np.float64))
    bad = np.abs(g - r) > 1e-2 + 2e-2 * scale
    assert not bad.any(), "%s: %d / %d outside the bound" % (what, bad.sum(), bad.size)


def test_calibrate_stack_teacher_forced():
    """The calibration pass of a stack on the residual map (Section III-B on
    the inputs each layer sees): at every layer, from the GPU's own inputs,
    the router logits, the layer output added to the residual stream and the
    next RMSNorm match the oracle; the similarity of each layer matches the
    oracle's on that layer's inputs; the counts of Eq. 5 add up and differ
    only at near ties; the transitions of Eq. 41 are bit for bit the oracle's
    on the recorded logits."""
    from paper_2607_17154_gb300.layer import calibrate_stack
    L, N, E, d, dff, k, M = 4, 1500, 8, 512, 512, 2, 4
    layers, hb = [], []
    for l in range(L):
        W1, W3, W2 = synth.ffn_weights(E, d, dff, seed=300 + l, device=DEV)
        layers.append({"W_r": synth.router_weights(E, d, 4, seed=310 + l, device=DEV),
                       "W1": W1, "W3": W3, "W2": W2})
    h_cal = synth.calibration(N, d, 320, device=DEV)
    cal = calibrate_stack(layers, h_cal, k, M)
    torch.cuda.synchronize()
    xs = [synth.bits(x) for x in cal["xs"]]
    hs = [synth.bits(h) for h in cal["hs"]]
    logits = cal["logits"].cpu().numpy()
    sim = cal["sim"].cpu().numpy()
    counts = cal["counts"].cpu().numpy()
    assert_norm_close(xs[0], oracle.rmsnorm(hs[0], EPS), "x_0")
    for l in range(L):
        lay = {n: synth.bits(t) for n, t in layers[l].items()}
        np.testing.assert_allclose(logits[l], oracle.router_logits(xs[l], lay["W_r"]), rtol=1e-3,
                                   atol=2e-3)
        idx, w = oracle.topk(logits[l], k)        # the unmodified model: every routed expert runs
        _, Y = oracle.ffn_rows(np.repeat(xs[l], k, axis=0), idx.reshape(-1), lay["W1"], lay["W3"],
                               lay["W2"])
        ref = oracle.combine_residual(Y, np.arange(N * k, dtype=np.int32).reshape(N, k), w, hs[l])
        _close_residual(hs[l + 1], ref, hs[l], w, Y.reshape(N, k, d), "h_%d" % (l + 1))
        assert_norm_close(xs[l + 1], oracle.rmsnorm(hs[l + 1], EPS), "x_%d" % (l + 1))
        o_sim, H = oracle.similarity(lay["W_r"], xs[l], return_H=True)
        np.testing.assert_allclose(sim[l], o_sim, atol=2e-5)
        o_counts = oracle.expert_counts(np.ascontiguousarray(H.T), k)
        srt = -np.sort(-H.T.astype(np.float64), axis=1)
        near = int((np.abs(srt[:, k - 1] - srt[:, k]) < 1e-3).sum())
        assert counts[l].sum() == N * k
        assert np.abs(counts[l] - o_counts).sum() <= 2 * near
    ref_c, ref_P = oracle.transitions(np.ascontiguousarray(logits.transpose(1, 0, 2)), k)
    np.testing.assert_array_equal(cal["tcount"].cpu().numpy(), ref_c)
    np.testing.assert_array_equal(cal["P"].cpu().numpy().view(np.uint32), ref_P.view(np.uint32))
