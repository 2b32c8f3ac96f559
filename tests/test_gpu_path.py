"""GPU parity of the hot path (router, selection, permutation, expert FFN,
combine) against the CPU oracle, through the C ABI."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_17154_gb300 import binding as B
from paper_2607_17154_gb300 import synth
from paper_2607_17154_gb300.layer import MoELayer, build_tables
from tests.helpers import (assert_close_bf16, assert_close_combined, check_layer_integers_full,
                           oracle_plan)

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


def dev(a, dtype=None):
    t = torch.as_tensor(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.to(dtype)
    return t.to(DEV)


def bf(bits):
    return synth.from_bits(bits).to(DEV)


def gbits(t):
    return synth.bits(t)


def random_tables_case(rng, E, M, n_groups):
    Wt = rng.standard_normal((E, 8))
    Wt[:, 0] += 3.0 * (np.arange(E) % n_groups)
    nrm = np.linalg.norm(Wt, axis=1, keepdims=True)
    sim = ((Wt / nrm) @ (Wt / nrm).T).astype(np.float32)
    np.fill_diagonal(sim, 1.0)
    group = (np.arange(E) % n_groups).astype(np.int32)
    x = (rng.random((M, E)) < 0.35).astype(np.uint8)
    for e in range(E):
        if not x[:, e].any():
            x[rng.integers(M), e] = 1
    return sim, group, x


# ------------------------------------------------------------------ tables

@pytest.mark.parametrize("E,M", [(8, 4), (64, 8), (5, 3), (64, 32)])
def test_tables_bit_exact(E, M):
    rng = np.random.default_rng(E * 100 + M)
    sim, group, x = random_tables_case(rng, E, M, 4)
    sp = synth.server_params(M, 4096, 14336, seed=E + M)
    for theta, qbar in [(0.5, 0.05), (-1.0, 0.3), (0.9, 0.0)]:
        t = build_tables(sim, group, x, theta, qbar, sp, DEV).cpu().numpy()
        ref = oracle.tables(sim, group, x, theta, qbar, sp.F, sp.B, sp.tau, sp.z, sp.c,
                            sp.omega_T, sp.omega_Q)
        hdr = t[:64].view(np.int32)
        assert hdr[0] == 0x4f4d5442 and hdr[1] == E and hdr[2] == M
        np.testing.assert_array_equal(t[64:64 + 4 * E].view(np.uint32), ref.pmask)
        np.testing.assert_array_equal(t[320:320 + 8 * E].view(np.uint64), ref.subst)
        o = 832
        np.testing.assert_array_equal(t[o:o + 4 * E * E].view(np.float32).reshape(E, E), ref.Qtab)
        o += 4 * E * E
        np.testing.assert_array_equal(t[o:o + 4 * E * E].view(np.float32).reshape(E, E), ref.Cq)
        o += 4 * E * E
        np.testing.assert_array_equal(t[o:o + 4 * M ** 3].view(np.float32).reshape(M, M, M), ref.A)


# ------------------------------------------------------------------ selection

@pytest.mark.parametrize("T,E,M,k", [(64, 8, 4, 2), (1000, 64, 8, 6), (37, 5, 3, 3), (300, 16, 32, 8)])
def test_route_select_given_logits_bit_exact(T, E, M, k):
    """Fed the same fp32 logits, top-k and every selection output match the
    oracle bit for bit (weights to 1e-5)."""
    rng = np.random.default_rng(T + E)
    sim, group, x = random_tables_case(rng, E, M, max(1, E // 8))
    sp = synth.server_params(M, 2048, 1408, seed=7)
    if E == 5:
        sp.tau[:] *= 1e-4                    # cheap links: remote candidates compete
    logits = rng.standard_normal((T, E)).astype(np.float32)
    logits[0, :] = 0.25                      # all tied
    home = rng.integers(0, M, T).astype(np.uint8)
    loc = np.where(rng.random(T) < 0.6, home, rng.integers(0, M, T)).astype(np.uint8)
    for theta, qbar in [(0.3, 0.1), (0.7, 0.05), (-1.0, 1.0)]:
        qhat = (rng.random(T) * qbar * 0.5).astype(np.float32)
        tab = build_tables(sim, group, x, theta, qbar, sp, DEV)
        o_idx, o_w = oracle.topk(logits, k, 1)
        o_tab = oracle.tables(sim, group, x, theta, qbar, sp.F, sp.B, sp.tau, sp.z, sp.c,
                              sp.omega_T, sp.omega_Q)
        och, osv, okd, oloc, oq = oracle.select(o_idx, o_tab, home, loc, qhat)
        g = dict(idx=torch.empty(T, k, dtype=torch.int32, device=DEV),
                 w=torch.empty(T, k, dtype=torch.float32, device=DEV),
                 ch=torch.empty(T, k, dtype=torch.int32, device=DEV),
                 sv=torch.empty(T, k, dtype=torch.uint8, device=DEV),
                 kd=torch.empty(T, k, dtype=torch.uint8, device=DEV),
                 cnt=torch.zeros(4, dtype=torch.int32, device=DEV))
        gloc = dev(loc); gq = dev(qhat)
        B.ordermoe_route_select(None, None, dev(logits), T, E, 0, k, 1, tab, dev(home), gloc, gq,
                                None, g["idx"], g["w"], g["ch"], g["sv"], g["kd"], g["cnt"])
        np.testing.assert_array_equal(g["idx"].cpu().numpy(), o_idx)
        np.testing.assert_allclose(g["w"].cpu().numpy(), o_w, rtol=1e-5, atol=1e-7)
        np.testing.assert_array_equal(g["ch"].cpu().numpy(), och)
        np.testing.assert_array_equal(g["sv"].cpu().numpy(), osv)
        np.testing.assert_array_equal(g["kd"].cpu().numpy(), okd)
        np.testing.assert_array_equal(gloc.cpu().numpy(), oloc)
        np.testing.assert_array_equal(gq.cpu().numpy(), oq)
        np.testing.assert_array_equal(g["cnt"].cpu().numpy(), np.bincount(okd.ravel(), minlength=4))


@pytest.mark.parametrize("T,d,E", [(300, 1024, 8), (600, 1024, 8), (100, 2048, 16), (700, 512, 16),
                                   (200, 256, 64), (512, 4096, 8), (513, 4096, 8)])
def test_router_logits_match_oracle(T, d, E):
    """The tcgen05 router (one to five 128-row tiles, split-K clusters, E up to
    64) against the oracle's logits, and the decisions taken from the GPU's
    own logits."""
    w = synth.workload("tiny", T=T, d=d, E=E, n_clusters=2)
    inp = synth.layer_inputs(w, seed=3, with_ffn=False)
    Xb, Wb = gbits(inp["X"]), gbits(inp["Wr"])
    ref = oracle.router_logits(Xb, Wb)
    E, M, k, T = w.E, w.M, w.k, w.T
    sim, group, x = random_tables_case(np.random.default_rng(0), E, M, 2)
    tab = build_tables(sim, group, x, 0.5, 0.05, synth.server_params(M, w.d, w.dff, 0), DEV)
    logits = torch.empty(T, E, dtype=torch.float32, device=DEV)
    outs = [torch.empty(T, k, dtype=dt, device=DEV)
            for dt in (torch.int32, torch.float32, torch.int32, torch.uint8, torch.uint8)]
    home = dev(inp["home"])
    B.ordermoe_route_select(inp["X"].to(DEV), inp["Wr"].to(DEV), None, T, E, w.d, k, 1, tab, home,
                            home.clone(), torch.zeros(T, device=DEV), logits, *outs)
    got = logits.cpu().numpy()
    np.testing.assert_allclose(got, ref, rtol=1e-3, atol=2e-3)
    # top-k and selection from the GPU's own logits equal the oracle's on the same logits
    o_idx, _ = oracle.topk(got, k, 1)
    np.testing.assert_array_equal(outs[0].cpu().numpy(), o_idx)
    sp = synth.server_params(M, w.d, w.dff, 0)
    otab = oracle.tables(sim, group, x, 0.5, 0.05, sp.F, sp.B, sp.tau, sp.z, sp.c, sp.omega_T,
                         sp.omega_Q)
    h = inp["home"]
    ch, sv, kd, _, _ = oracle.select(o_idx, otab, h, h.copy(), np.zeros(T, np.float32))
    np.testing.assert_array_equal(outs[2].cpu().numpy(), ch)
    np.testing.assert_array_equal(outs[3].cpu().numpy(), sv)
    np.testing.assert_array_equal(outs[4].cpu().numpy(), kd)


@pytest.mark.parametrize("E,k", [(8, 1), (13, 3), (16, 5), (16, 7), (16, 8), (24, 3), (32, 4),
                                 (40, 6), (64, 2), (64, 6), (64, 8)])
def test_router_exact_ties_every_list_width(E, k):
    """Router rows copied in groups of 2 and 3 alternately (each row of a group
    equal to the group's first), so every logit the tensor-core router
    computes has bitwise-equal siblings and, for every k, equal logits
    straddle the k-th rank for some tokens: the top-k (a sorted list of 2, 4,
    6 or 8 entries; E not a multiple of 4 padded with -inf) must keep the lower
    index first, as the oracle does on the GPU's own logits (Alg. 2's
    targets), and the selection from those targets must match bit for bit."""
    T, d = 300, 512
    w = synth.workload("tiny", T=T, d=d, E=E, n_clusters=1)
    inp = synth.layer_inputs(w, seed=9, with_ffn=False)
    lead, r, size = np.arange(E), 0, 2
    while r < E:
        lead[r:r + size] = r
        r, size = r + size, 5 - size
    Wr = inp["Wr"][torch.as_tensor(lead)].contiguous()
    M = w.M
    sim, group, x = random_tables_case(np.random.default_rng(E + k), E, M, 2)
    tab = build_tables(sim, group, x, 0.5, 0.05, synth.server_params(M, d, w.dff, 0), DEV)
    logits = torch.empty(T, E, dtype=torch.float32, device=DEV)
    outs = [torch.empty(T, k, dtype=dt, device=DEV)
            for dt in (torch.int32, torch.float32, torch.int32, torch.uint8, torch.uint8)]
    home = dev(inp["home"])
    B.ordermoe_route_select(inp["X"].to(DEV), Wr.to(DEV), None, T, E, d, k, 1, tab, home,
                            home.clone(), torch.zeros(T, device=DEV), logits, *outs)
    got = logits.cpu().numpy()
    np.testing.assert_array_equal(got, got[:, lead])
    np.testing.assert_allclose(got, oracle.router_logits(gbits(inp["X"]), gbits(Wr)), rtol=1e-3,
                               atol=2e-3)
    o_idx, o_w = oracle.topk(got, k, 1)
    np.testing.assert_array_equal(outs[0].cpu().numpy(), o_idx)
    np.testing.assert_allclose(outs[1].cpu().numpy(), o_w, rtol=1e-5, atol=1e-7)
    # a tie at the boundary: the k-th and (k + 1)-th logits equal for some token
    srt = -np.sort(-got, axis=1)
    assert (srt[:, k - 1] == srt[:, k]).any()
    sp = synth.server_params(M, d, w.dff, 0)
    otab = oracle.tables(sim, group, x, 0.5, 0.05, sp.F, sp.B, sp.tau, sp.z, sp.c, sp.omega_T,
                         sp.omega_Q)
    h = inp["home"]
    ch, sv, kd, _, _ = oracle.select(o_idx, otab, h, h.copy(), np.zeros(T, np.float32))
    np.testing.assert_array_equal(outs[2].cpu().numpy(), ch)
    np.testing.assert_array_equal(outs[3].cpu().numpy(), sv)
    np.testing.assert_array_equal(outs[4].cpu().numpy(), kd)


# ------------------------------------------------------------------ permutation

@pytest.mark.parametrize("T,k,E,d", [(64, 2, 8, 256), (1000, 6, 64, 64), (1, 1, 1, 8), (333, 3, 7, 40),
                                     # one block ranking several rounds of 1024 entries, up to
                                     # its limit of 4096, and the first size past it
                                     (1500, 2, 8, 64), (2048, 2, 8, 16), (683, 6, 64, 8),
                                     (4096, 2, 8, 4096),
                                     (8192, 6, 64, 64),     # 192 chunks: the scan holds them in registers
                                     (16384, 4, 64, 64),    # 256 chunks: the most it holds in registers
                                     (16385, 4, 33, 64),    # 257 chunks: 32 at a time from memory
                                     (20000, 6, 64, 64)])   # 469 chunks x 64
def test_dispatch_bit_exact(T, k, E, d):
    rng = np.random.default_rng(T * k + E)
    chosen = rng.integers(0, E, (T, k)).astype(np.int32)
    if E > 2:
        chosen[chosen == 1] = 0              # an expert with no rows
    X = synth.normal((T, d), 1.0, seed=T)
    off, rt, rof = oracle.dispatch(chosen, E)
    Xp_ref = oracle.gather_rows(gbits(X), rt)
    g_off = torch.empty(E + 1, dtype=torch.int32, device=DEV)
    g_rt = torch.empty(T * k, dtype=torch.int32, device=DEV)
    g_rof = torch.empty(T, k, dtype=torch.int32, device=DEV)
    g_xp = torch.empty(T * k, d, dtype=torch.bfloat16, device=DEV)
    ws = torch.empty(B.ordermoe_dispatch_workspace_bytes(T, k, E), dtype=torch.uint8, device=DEV)
    B.ordermoe_dispatch(dev(chosen), X.to(DEV), T, k, E, d, g_off, g_rt, g_rof, g_xp, ws)
    np.testing.assert_array_equal(g_off.cpu().numpy(), off)
    np.testing.assert_array_equal(g_rt.cpu().numpy(), rt)
    np.testing.assert_array_equal(g_rof.cpu().numpy(), rof)
    np.testing.assert_array_equal(gbits(g_xp), Xp_ref)


def test_dispatch_empty():
    E = 4
    g_off = torch.full((E + 1,), 7, dtype=torch.int32, device=DEV)
    z = torch.empty(0, dtype=torch.int32, device=DEV)
    B.ordermoe_dispatch(z.view(0, 2), torch.empty(0, 64, dtype=torch.bfloat16, device=DEV), 0, 2, E,
                        64, g_off, z, z.view(0, 2), torch.empty(0, 64, dtype=torch.bfloat16, device=DEV),
                        torch.empty(256, dtype=torch.uint8, device=DEV))
    assert (g_off.cpu().numpy() == 0).all()


# ------------------------------------------------------------------ expert FFN

def ffn_case(rows_per_expert, d, dff, seed):
    E = len(rows_per_expert)
    R = int(sum(rows_per_expert))
    off = np.concatenate([[0], np.cumsum(rows_per_expert)]).astype(np.int32)
    row_e = np.repeat(np.arange(E), rows_per_expert).astype(np.int32)
    Xp = synth.normal((R, d), 1.0, seed)
    W1, W3, W2 = synth.ffn_weights(E, d, dff, seed + 1)
    return E, R, off, row_e, Xp, W1, W3, W2


def run_gpu_ffn(E, R, off, Xp, W1, W3, W2, d, dff):
    H = torch.zeros(R, dff, dtype=torch.bfloat16, device=DEV)
    Y = torch.zeros(R, d, dtype=torch.bfloat16, device=DEV)
    B.ordermoe_expert_ffn(Xp.to(DEV), dev(off), R, W1.to(DEV), W3.to(DEV), W2.to(DEV), E, d, dff, H, Y)
    torch.cuda.synchronize()
    return H, Y


@pytest.mark.parametrize("rows,d,dff", [
    ([16, 16, 16, 16, 16, 16, 16, 16], 256, 512),         # tiny layer, one partial tile each
    ([300, 0, 1, 128, 129, 77], 512, 384),                # ragged tails, empty and 1-row experts
    ([37], 256, 128),                                     # one partial tile
    ([256, 256], 1024, 1024),                             # several full tiles and K blocks
    # CTA pairs (at least 256 rows per expert on average): last row tiles of
    # 1, 128, 88, 44, 1, 129 and 255 rows, cut to N = 16, 128, 96, 48, 16, 144
    # and 256 columns of the transposed accumulator
    ([257, 384, 600, 300, 512, 1], 256, 512),
    ([129, 255, 256, 384], 512, 384),
])
def test_expert_ffn_matches_oracle(rows, d, dff):
    E, R, off, row_e, Xp, W1, W3, W2 = ffn_case(rows, d, dff, seed=sum(rows) + d)
    H, Y = run_gpu_ffn(E, R, off, Xp, W1, W3, W2, d, dff)
    Href, Yref = oracle.ffn_rows(gbits(Xp), row_e, gbits(W1), gbits(W3), gbits(W2))
    assert_close_bf16(gbits(H), Href, what="H")
    assert_close_bf16(gbits(Y), Yref, what="Y")


# ------------------------------------------------------------------ combine

@pytest.mark.parametrize("T,k,d", [(64, 2, 256), (513, 6, 2048), (5, 8, 8)])
def test_combine_matches_oracle(T, k, d):
    rng = np.random.default_rng(T + k)
    Yp = synth.normal((T * k, d), 1.0, seed=T)
    row_of = rng.permutation(T * k).astype(np.int32).reshape(T, k)
    w = rng.random((T, k)).astype(np.float32)
    y = torch.empty(T, d, dtype=torch.bfloat16, device=DEV)
    B.ordermoe_combine(Yp.to(DEV), dev(row_of), dev(w), T, k, d, y)
    ref = oracle.combine(gbits(Yp), row_of, w)
    assert_close_bf16(gbits(y), ref, rtol=1e-2, atol=1e-3, what="y")


# ------------------------------------------------------------------ whole layer

def layer_setup(w, seed, device_gen="cpu"):
    inp = synth.layer_inputs(w, seed=seed)
    Xcal = synth.calibration(w.n_cal, w.d, seed)
    plan = oracle_plan(gbits(inp["Wr"]), gbits(Xcal), w.k, w.M, w.theta)
    sp = synth.server_params(w.M, w.d, w.dff, seed)
    return inp, plan, sp


def layer_gpu_arrays(layer, T, loc, qhat, with_xperm=True):
    """Host copies of one MoELayer call's integer outputs (and X_perm bits)."""
    R = T * layer.k
    out = {"idx": layer.topk_idx[:T].cpu().numpy(), "w": layer.topk_w[:T].cpu().numpy(),
           "chosen": layer.chosen[:T].cpu().numpy(), "server": layer.server[:T].cpu().numpy(),
           "kind": layer.kind[:T].cpu().numpy(), "loc": loc[:T].cpu().numpy(),
           "qhat": qhat[:T].cpu().numpy(), "offsets": layer.offsets.cpu().numpy(),
           "row_token": layer.row_token[:R].cpu().numpy(), "row_of": layer.row_of[:T].cpu().numpy()}
    if with_xperm:
        out["X_perm"] = gbits(layer.X_perm[:R])
    return out


def run_layer_check(w, seed, sample=None):
    """One layer at the workload's full size.

    * Every integer output over ALL T tokens, near ties included, bit for bit:
      the oracle's top-k, selection (Eqs. 40, 43, 44) and permutation run on
      the GPU's own fp32 router logits (the same numbers on both sides).
    * Router logits of the sampled tokens against the oracle's fp64 sums, and
      the oracle's own decisions from its own logits wherever the top-k is
      unambiguous at that precision.
    * Expert outputs Y and the combined y of the sampled tokens (all of them,
      near ties included) against the oracle's FFN and combine of the same
      decisions, within rtol 2e-2 / atol 1e-2."""
    inp, plan, sp = layer_setup(w, seed)
    tab = build_tables(plan["sim"], plan["group"], plan["placement"], w.theta, w.qbar, sp, DEV)
    g = {n: inp[n].to(DEV) for n in ("X", "Wr", "W1", "W3", "W2")}
    layer = MoELayer(g["Wr"], g["W1"], g["W3"], g["W2"], tab, w.k, w.T)
    home = dev(inp["home"]); loc = home.clone(); qhat = torch.zeros(w.T, device=DEV)
    y = torch.empty(w.T, w.d, dtype=torch.bfloat16, device=DEV)
    layer.forward(g["X"], home, loc, qhat, y)
    torch.cuda.synchronize()
    o_tab = oracle.tables(plan["sim"], plan["group"], plan["placement"], w.theta, w.qbar, sp.F, sp.B,
                          sp.tau, sp.z, sp.c, sp.omega_T, sp.omega_Q)
    h = inp["home"]
    Xb = gbits(inp["X"])
    g_logits_all = layer.logits.cpu().numpy()
    gpu = layer_gpu_arrays(layer, w.T, loc, qhat)
    idx, wt, chosen = check_layer_integers_full(g_logits_all, gpu, o_tab, h, h,
                                                np.zeros(w.T, np.float32), w.k, w.E, X_bits=Xb,
                                                what=w.name)
    toks = np.arange(w.T) if sample is None else np.sort(
        np.random.default_rng(seed).choice(w.T, sample, replace=False))
    # Router logits: fp32 tensor-core sums vs the oracle's fp64 sums.
    o_logits = oracle.router_logits(np.ascontiguousarray(Xb[toks]), gbits(inp["Wr"]))
    g_logits = g_logits_all[toks]
    np.testing.assert_allclose(g_logits, o_logits, rtol=1e-3, atol=2e-3)
    # The oracle's decisions from its own logits agree wherever every gap
    # around the k-th rank exceeds the logit disagreement (8x the largest one
    # seen); near ties there are covered by the full check above.
    delta = max(8.0 * float(np.abs(g_logits - o_logits).max()), 1e-6)
    srt = -np.sort(-o_logits.astype(np.float64), axis=1)
    margin = np.abs(np.diff(srt[:, :min(w.k + 1, w.E)], axis=1)).min(axis=1)
    clear = margin > delta
    assert clear.mean() > 0.5, (clear.mean(), delta)
    oidx, _ = oracle.topk(o_logits, w.k)
    och, osv, okd, oloc, oq = oracle.select(oidx, o_tab, h[toks], h[toks].copy(),
                                            np.zeros(len(toks), np.float32))
    for name, ref in (("idx", oidx), ("chosen", och), ("server", osv), ("kind", okd)):
        np.testing.assert_array_equal(gpu[name][toks][clear], ref[clear], err_msg=name)
    np.testing.assert_array_equal(gpu["loc"][toks][clear], oloc[clear])
    # expert outputs and combine of every sampled token, from the decisions
    # checked above
    rows = np.repeat(np.ascontiguousarray(Xb[toks]), w.k, axis=0)
    _, Yref = oracle.ffn_rows(rows, chosen[toks].reshape(-1).astype(np.int32), gbits(inp["W1"]),
                              gbits(inp["W3"]), gbits(inp["W2"]))
    n = len(toks)
    Yref = Yref.reshape(n, w.k, -1)
    yref = oracle.combine(Yref.reshape(n * w.k, -1), np.arange(n * w.k, dtype=np.int32).reshape(n, w.k),
                          wt[toks])
    Yg = gbits(layer.Y_perm)[gpu["row_of"][toks]]          # [n, k, d]
    assert_close_bf16(Yg, Yref, what="expert outputs Y")
    assert_close_combined(gbits(y)[toks], yref, wt[toks], Yref)
    return layer


def test_layer_tiny_all_tokens():
    w = synth.workload("tiny")
    layer = run_layer_check(w, seed=0)
    kinds = layer.counters.cpu().numpy()
    assert kinds.sum() == w.T * w.k


def test_layer_fine_grained_shape_sampled():
    w = synth.workload("fine_grained", T=2048)
    run_layer_check(w, seed=1, sample=96)


def test_layer_mixtral_prefill_full_size_sampled():
    w = synth.workload("mixtral_prefill")
    run_layer_check(w, seed=0, sample=512)


# ------------------------------------------------------------------ errors and bounded waits

def test_host_side_argument_errors():
    z8 = torch.zeros(64, dtype=torch.uint8, device=DEV)
    with pytest.raises(B.OrderMoEError) as ei:
        B.ordermoe_expert_ffn(*(torch.zeros(128, 100, dtype=torch.bfloat16, device=DEV),
                                torch.zeros(3, dtype=torch.int32, device=DEV), 128,
                                torch.zeros(2, 128, 100, dtype=torch.bfloat16, device=DEV),
                                torch.zeros(2, 128, 100, dtype=torch.bfloat16, device=DEV),
                                torch.zeros(2, 100, 128, dtype=torch.bfloat16, device=DEV),
                                2, 100, 128,
                                torch.zeros(128, 128, dtype=torch.bfloat16, device=DEV),
                                torch.zeros(128, 100, dtype=torch.bfloat16, device=DEV)))
    assert ei.value.code == B.ERR_UNSUPPORTED_SHAPE
    with pytest.raises(B.OrderMoEError) as ei:
        B.ordermoe_route_select(None, None, torch.zeros(4, 8, device=DEV), 4, 8, 0, 9, 1, z8,
                                z8[:4], z8[:4], torch.zeros(4, device=DEV), None,
                                *[torch.zeros(4, 9, dtype=dt, device=DEV) for dt in
                                  (torch.int32, torch.float32, torch.int32, torch.uint8, torch.uint8)])
    assert ei.value.code == B.ERR_UNSUPPORTED_SHAPE


def test_nan_logit_sets_device_error():
    E, M, T, k = 8, 4, 8, 2
    sim, group, x = random_tables_case(np.random.default_rng(1), E, M, 2)
    tab = build_tables(sim, group, x, 0.5, 0.1, synth.server_params(M, 256, 512, 0), DEV)
    logits = torch.zeros(T, E, device=DEV); logits[3, 2] = float("nan")
    home = torch.zeros(T, dtype=torch.uint8, device=DEV)
    outs = [torch.empty(T, k, dtype=dt, device=DEV)
            for dt in (torch.int32, torch.float32, torch.int32, torch.uint8, torch.uint8)]
    B.ordermoe_route_select(None, None, logits, T, E, 0, k, 1, tab, home, home.clone(),
                            torch.zeros(T, device=DEV), None, *outs)
    code, detail = B.ordermoe_device_error()
    assert code == B.DEV_NAN_LOGIT and detail == 3


def test_bounded_wait_runs_out_and_reports():
    B.ordermoe_selftest_wait_timeout(2_000_000)          # 2 ms, nothing ever arrives
    code, detail = B.ordermoe_device_error()
    assert code == B.DEV_WAIT_TIMEOUT and detail == 99
    # the context is still usable afterwards
    x = torch.ones(16, device=DEV)
    assert float(x.sum()) == 16.0


def test_bad_row_index_in_combine_is_reported_not_read():
    T, k, d = 16, 2, 64
    Yp = torch.zeros(T * k, d, dtype=torch.bfloat16, device=DEV)
    row_of = torch.arange(T * k, dtype=torch.int32, device=DEV).view(T, k).clone()
    row_of[5, 1] = T * k + 1000                      # outside Y_perm
    y = torch.full((T, d), 7.0, dtype=torch.bfloat16, device=DEV)
    B.ordermoe_combine(Yp, row_of, torch.ones(T, k, device=DEV), T, k, d, y)
    code, detail = B.ordermoe_device_error()
    assert code == B.DEV_BAD_INDEX and detail == 5
    yc = y.cpu().float()
    assert (yc[5] == 7.0).all() and (yc[4] == 0).all()


def test_bad_offsets_in_expert_ffn_are_reported_not_used():
    E, R, d, dff = 3, 64, 256, 128
    z = lambda *s: torch.zeros(*s, dtype=torch.bfloat16, device=DEV)
    W1, W3, W2 = z(E, dff, d), z(E, dff, d), z(E, d, dff)
    H = torch.full((R, dff), 3.0, dtype=torch.bfloat16, device=DEV)
    Y = torch.full((R, d), 3.0, dtype=torch.bfloat16, device=DEV)
    for bad in ([0, 40, 20, 64], [0, 10, 20, 4000], [5, 10, 20, 64]):
        B.ordermoe_expert_ffn(z(R, d), torch.tensor(bad, dtype=torch.int32, device=DEV), R, W1, W3,
                              W2, E, d, dff, H, Y)
        code, detail = B.ordermoe_device_error()
        assert code == B.DEV_BAD_INDEX and detail == -2, bad
    assert (H.cpu().float() == 3.0).all() and (Y.cpu().float() == 3.0).all()
