"""Test-side helpers: run the oracle's offline plan (Eqs. 3-6, 24-31) and the
oracle's per-token forward for sampled tokens."""
import numpy as np

import oracle
from paper_2607_17154_gb300 import synth


def bits_to_f(b):
    return (np.asarray(b, np.uint16).astype(np.uint32) << 16).view(np.float32)


def oracle_plan(Wr_bits, Xcal_bits, k, M, theta, p_unit=1.0):
    """Similarity, counts, groups and placement of one layer by the oracle."""
    E = Wr_bits.shape[0]
    sim, H = oracle.similarity(Wr_bits, Xcal_bits, return_H=True)
    counts = oracle.expert_counts(np.ascontiguousarray(H.T), k)
    group, K, _ = oracle.group(sim, counts, theta)
    imp = oracle.importance(sim, counts, group)
    p = np.full((1, E), p_unit)
    C = np.full(M, E * p_unit / M)
    x, used, rc = oracle.place(group[None], imp[None], p, C)
    assert rc == 0
    return dict(sim=sim, counts=counts, group=group, K=K, placement=x[0])


def oracle_layer_tokens(tokens, X_bits, Wr_bits, W1, W3, W2, tab, home, loc, qhat, k, renorm=1):
    """Oracle forward of the listed tokens through one layer.

    Returns (y [n,d] bf16 bits, idx, w, chosen, server, kind, margin) where
    margin is the oracle's logit gap around the k-th rank (small = near tie)."""
    Xs = X_bits[tokens]
    logits = oracle.router_logits(Xs, Wr_bits)
    idx, w = oracle.topk(logits, k, renorm)
    chosen, server, kind, loc2, q2 = oracle.select(idx, tab, home[tokens], loc[tokens], qhat[tokens])
    srt = -np.sort(-logits.astype(np.float64), axis=1)
    E = logits.shape[1]
    gaps = np.abs(np.diff(srt[:, :min(k + 1, E)], axis=1))
    margin = gaps.min(axis=1) if gaps.shape[1] else np.full(len(tokens), np.inf)
    n = len(tokens)
    rows = np.repeat(Xs, k, axis=0)
    _, Y = oracle.ffn_rows(rows, chosen.reshape(-1).astype(np.int32), W1, W3, W2)
    row_of = np.arange(n * k, dtype=np.int32).reshape(n, k)
    y = oracle.combine(Y, row_of, w)
    return dict(y=y, Y=Y.reshape(n, k, -1), logits=logits, idx=idx, w=w, chosen=chosen,
                server=server, kind=kind, loc=loc2, qhat=q2, margin=margin)


def assert_close_bf16(got_bits, ref_bits, rtol=2e-2, atol=1e-2, what=""):
    g = bits_to_f(got_bits).astype(np.float64)
    r = bits_to_f(ref_bits).astype(np.float64)
    bad = np.abs(g - r) > atol + rtol * np.abs(r)
    if bad.any():
        i = np.argwhere(bad)[:5]
        raise AssertionError("%s: %d / %d elements outside rtol=%g atol=%g; first %s: got %s ref %s"
                             % (what, bad.sum(), bad.size, rtol, atol, i.tolist(),
                                g[tuple(i.T)].tolist(), r[tuple(i.T)].tolist()))


def assert_close_combined(got_bits, ref_bits, w, Yref_bits, rtol=2e-2, atol=1e-2, what="y"):
    """Weighted-sum check: y = sum_j w_j Y_j is compared with a tolerance that
    scales with sum_j |w_j| |Y_j| (the magnitude the rounding of each Y_j
    carries into y), since the slots can cancel."""
    g = bits_to_f(got_bits).astype(np.float64)
    r = bits_to_f(ref_bits).astype(np.float64)
    scale = np.einsum("tk,tkd->td", np.abs(w).astype(np.float64),
                      np.abs(bits_to_f(Yref_bits).astype(np.float64)))
    bad = np.abs(g - r) > atol + rtol * scale
    if bad.any():
        i = np.argwhere(bad)[:5]
        raise AssertionError("%s: %d / %d elements outside the combine bound; first %s: got %s ref %s"
                             % (what, bad.sum(), bad.size, i.tolist(), g[tuple(i.T)].tolist(),
                                r[tuple(i.T)].tolist()))


def check_layer_integers_full(logits, gpu, o_tab, home, loc_in, qhat_in, k, E, X_bits=None,
                              renorm=1, what=""):
    """Bit-exact parity of every integer decision of one layer over ALL its
    tokens, near ties included: the oracle's top-k (Alg. 2's target), the
    selection of Eqs. 40, 43, 44 and the permutation are run on the GPU's own
    fp32 router logits, so both sides decide from the same numbers.

    gpu: dict of host arrays from the GPU (idx, w, chosen, server, kind, loc,
    qhat, and optionally offsets, row_token, row_of, X_perm bits).
    Returns the oracle's (idx, w, chosen) for reuse."""
    logits = np.ascontiguousarray(logits, np.float32)
    idx, w = oracle.topk(logits, k, renorm)
    np.testing.assert_array_equal(gpu["idx"], idx, err_msg=what + " top-k idx")
    np.testing.assert_allclose(gpu["w"], w, rtol=1e-5, atol=1e-7, err_msg=what + " gate weights")
    chosen, server, kind, loc2, q2 = oracle.select(idx, o_tab, np.asarray(home, np.uint8),
                                                   np.array(loc_in, np.uint8, copy=True),
                                                   np.array(qhat_in, np.float32, copy=True))
    for name, ref in (("chosen", chosen), ("server", server), ("kind", kind), ("loc", loc2)):
        np.testing.assert_array_equal(gpu[name], ref, err_msg="%s %s" % (what, name))
    # the accumulated loss compared as bits (Eq. 44's fp32 adds in slot order)
    np.testing.assert_array_equal(np.asarray(gpu["qhat"], np.float32).view(np.uint32),
                                  q2.view(np.uint32), err_msg=what + " qhat")
    if "offsets" in gpu:
        off, rt, row_of = oracle.dispatch(chosen.astype(np.int32), E)
        np.testing.assert_array_equal(gpu["offsets"], off, err_msg=what + " offsets")
        np.testing.assert_array_equal(gpu["row_token"], rt, err_msg=what + " row_token")
        np.testing.assert_array_equal(gpu["row_of"], row_of, err_msg=what + " row_of")
        if X_bits is not None and "X_perm" in gpu:
            np.testing.assert_array_equal(gpu["X_perm"], oracle.gather_rows(X_bits, rt),
                                          err_msg=what + " X_perm")
    return idx, w, chosen
