"""Python access to the OrderMoE CPU oracle (numpy in, numpy out).

TEST INFRASTRUCTURE ONLY: the slow, plain reference that the CUDA library is
checked against. Only tests/, __graft_entry__.smoke() and the CPU-baseline
leg of bench.py may import this package. It shares no code with the CUDA
library (paper_2607_17154_gb300) and never imports it.

Every wrapper below forwards to the C++ function of the same stem in
ordermoe_oracle.cpp, which names the paper's section and equation it follows.
bf16 arrays travel as np.uint16 bit patterns.
"""
import ctypes
import os

import numpy as np

from . import build as _build

_lib = None

_P = ctypes.c_void_p
_I = ctypes.c_int
_I64 = ctypes.c_int64
_F = ctypes.c_float
_D = ctypes.c_double

OK, BAD_ARG, NAN, CAPACITY = 0, 1, 2, 3


class OracleError(RuntimeError):
    pass


def lib():
    global _lib
    if _lib is None:
        path = _build.build()
        L = ctypes.CDLL(path)
        sigs = {
            "orc_router_logits": [_P, _P, _I, _I, _I, _P],
            "orc_topk": [_P, _I, _I, _I, _I, _P, _P],
            "orc_tables": [_P, _P, _P, _I, _I, _F, _F, _P, _P, _P, _D, _D, _D, _D, _P, _P, _P, _P, _P],
            "orc_select": [_P, _I, _I, _I, _I, _P, _P, _P, _P, _P, _F, _P, _P, _P, _P, _P, _P],
            "orc_dispatch": [_P, _I, _I, _I, _P, _P, _P],
            "orc_gather_rows": [_P, _P, _I64, _I, _P],
            "orc_ffn_rows": [_P, _P, _I64, _P, _P, _P, _I, _I, _I, _P, _P],
            "orc_combine": [_P, _P, _P, _I, _I, _I, _P],
            "orc_rmsnorm": [_P, _I, _I, _D, _P],
            "orc_combine_residual": [_P, _P, _P, _P, _I, _I, _I, _P],
            "orc_similarity": [_P, _P, _I, _I, _I64, _P, _P],
            "orc_expert_counts": [_P, _I64, _I, _I, _P],
            "orc_group": [_P, _P, _I, _F, _P, _P, _P],
            "orc_importance": [_P, _P, _P, _I, _D, _D, _P],
            "orc_place": [_P, _P, _P, _I, _I, _I, _P, _D, _D, _P, _P],
            "orc_coverage": [_P, _P, _I, _I, _I, _P],
            "orc_replicate": [_P, _P, _P, _I, _I, _I, _P, _P, _P, _P, _P],
            "orc_trajectory_cost": [_P, _P, _P, _P, _I, _I, _I, _I, _I, _P, _P, _P, _D, _D, _P,
                                    _P, _P, _P],
            "orc_utility": [_P, _P, _P, _I, _D, _D, _D, _D, _P],
            "orc_transitions": [_P, _I64, _I, _I, _I, _P, _P],
            "orc_select_lookahead": [_P, _I, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P,
                                     _P, _F, _P, _P, _P, _P, _P, _P],
        }
        for name, args in sigs.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = _I
        L.orc_threads.argtypes = []
        L.orc_threads.restype = _I
        L.orc_set_threads.argtypes = [_I]
        L.orc_set_threads.restype = _I
        L.orc_theta.argtypes = [_I, _I, _D, _D, _D]
        L.orc_theta.restype = _F
        _lib = L
    return _lib


def _c(a, dtype):
    """Contiguous array of the given dtype (bf16 tensors: pass .view(np.uint16))."""
    a = np.ascontiguousarray(a, dtype=dtype)
    return a


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p)


def _check(rc, name):
    if rc != OK:
        raise OracleError("%s returned %d" % (name, rc))


def router_logits(X, W):
    """X [T,d] bf16 bits, W [E,d] bf16 bits -> logits [T,E] f32 (Eq. 3, fp64 sum)."""
    X = _c(X, np.uint16); W = _c(W, np.uint16)
    T, d = X.shape; E = W.shape[0]
    out = np.empty((T, E), np.float32)
    _check(lib().orc_router_logits(_ptr(X), _ptr(W), T, E, d, _ptr(out)), "orc_router_logits")
    return out


def topk(logits, k, renorm=1):
    logits = _c(logits, np.float32)
    T, E = logits.shape
    idx = np.empty((T, k), np.int32); w = np.empty((T, k), np.float32)
    _check(lib().orc_topk(_ptr(logits), T, E, k, int(renorm), _ptr(idx), _ptr(w)), "orc_topk")
    return idx, w


class Tables:
    """The oracle's own per-layer selection tables (see orc_tables)."""

    def __init__(self, Qtab, Cq, subst, A, pmask, qbar, E, M):
        self.Qtab, self.Cq, self.subst, self.A, self.pmask = Qtab, Cq, subst, A, pmask
        self.qbar, self.E, self.M = np.float32(qbar), E, M


def tables(sim, group, placement, theta, qbar, F, B, tau, z, c, omega_T, omega_Q):
    sim = _c(sim, np.float32); group = _c(group, np.int32); placement = _c(placement, np.uint8)
    E = sim.shape[0]; M = placement.shape[0]
    F = _c(F, np.float64); B = _c(B, np.float64); tau = _c(tau, np.float64)
    Qtab = np.empty((E, E), np.float32); Cq = np.empty((E, E), np.float32)
    subst = np.empty(E, np.uint64); A = np.empty((M, M, M), np.float32)
    pmask = np.empty(E, np.uint32)
    rc = lib().orc_tables(_ptr(sim), _ptr(group), _ptr(placement), E, M, float(theta), float(qbar),
                          _ptr(F), _ptr(B), _ptr(tau), float(z), float(c), float(omega_T),
                          float(omega_Q), _ptr(Qtab), _ptr(Cq), _ptr(subst), _ptr(A), _ptr(pmask))
    _check(rc, "orc_tables")
    return Tables(Qtab, Cq, subst, A, pmask, qbar, E, M)


def select(idx, tab, home, loc, qhat):
    """Alg. 2 (H = 1). Returns chosen, server, kind and the updated loc, qhat."""
    idx = _c(idx, np.int32); T, k = idx.shape
    home = _c(home, np.uint8); loc = _c(loc, np.uint8).copy(); qhat = _c(qhat, np.float32).copy()
    chosen = np.empty((T, k), np.int32); server = np.empty((T, k), np.uint8)
    kind = np.empty((T, k), np.uint8)
    rc = lib().orc_select(_ptr(idx), T, tab.E, k, tab.M, _ptr(tab.Qtab), _ptr(tab.Cq),
                          _ptr(tab.subst), _ptr(tab.A), _ptr(tab.pmask), float(tab.qbar),
                          _ptr(home), _ptr(loc), _ptr(qhat), _ptr(chosen), _ptr(server), _ptr(kind))
    _check(rc, "orc_select")
    return chosen, server, kind, loc, qhat


def dispatch(chosen, E):
    chosen = _c(chosen, np.int32); T, k = chosen.shape
    offsets = np.empty(E + 1, np.int32); row_token = np.empty(T * k, np.int32)
    row_of = np.empty((T, k), np.int32)
    _check(lib().orc_dispatch(_ptr(chosen), T, k, E, _ptr(offsets), _ptr(row_token), _ptr(row_of)),
           "orc_dispatch")
    return offsets, row_token, row_of


def gather_rows(X, row_token):
    X = _c(X, np.uint16); row_token = _c(row_token, np.int32)
    R = row_token.shape[0]; d = X.shape[1]
    out = np.empty((R, d), np.uint16)
    _check(lib().orc_gather_rows(_ptr(X), _ptr(row_token), R, d, _ptr(out)), "orc_gather_rows")
    return out


def ffn_rows(Xrows, row_expert, W1, W3, W2):
    """Rows with their expert -> (H [R,dff], Y [R,d]) as bf16 bits."""
    Xrows = _c(Xrows, np.uint16); row_expert = _c(row_expert, np.int32)
    W1 = _c(W1, np.uint16); W3 = _c(W3, np.uint16); W2 = _c(W2, np.uint16)
    R, d = Xrows.shape; E, dff, _ = W1.shape
    H = np.zeros((R, dff), np.uint16); Y = np.zeros((R, d), np.uint16)
    rc = lib().orc_ffn_rows(_ptr(Xrows), _ptr(row_expert), R, _ptr(W1), _ptr(W3), _ptr(W2),
                            E, d, dff, _ptr(H), _ptr(Y))
    _check(rc, "orc_ffn_rows")
    return H, Y


def combine(Yp, row_of, w):
    Yp = _c(Yp, np.uint16); row_of = _c(row_of, np.int32); w = _c(w, np.float32)
    T, k = row_of.shape; d = Yp.shape[1]
    y = np.empty((T, d), np.uint16)
    _check(lib().orc_combine(_ptr(Yp), _ptr(row_of), _ptr(w), T, k, d, _ptr(y)), "orc_combine")
    return y


def threads():
    """OpenMP threads the oracle's parallel loops use."""
    return int(lib().orc_threads())


def set_threads(n):
    _check(lib().orc_set_threads(int(n)), "orc_set_threads")


def rmsnorm(h, eps=1e-6):
    """x = RMSNorm(h) of the residual map between stacked layers (bf16 bits, fp64 math)."""
    h = _c(h, np.uint16); T, d = h.shape
    x = np.empty((T, d), np.uint16)
    _check(lib().orc_rmsnorm(_ptr(h), T, d, float(eps), _ptr(x)), "orc_rmsnorm")
    return x


def combine_residual(Yp, row_of, w, h):
    """h_out = bf16(h + sum_j w_j Y[row_of[t][j]]) (bf16 bits, fp64 math)."""
    Yp = _c(Yp, np.uint16); row_of = _c(row_of, np.int32); w = _c(w, np.float32)
    h = _c(h, np.uint16)
    T, k = row_of.shape; d = h.shape[1]
    out = np.empty((T, d), np.uint16)
    _check(lib().orc_combine_residual(_ptr(Yp), _ptr(row_of), _ptr(w), _ptr(h), T, k, d,
                                      _ptr(out)), "orc_combine_residual")
    return out


def similarity(W, Xc, return_H=False):
    W = _c(W, np.uint16); Xc = _c(Xc, np.uint16)
    E, d = W.shape; N = Xc.shape[0]
    sim = np.empty((E, E), np.float32)
    H = np.empty((E, N), np.float32) if return_H else None
    rc = lib().orc_similarity(_ptr(W), _ptr(Xc), E, d, N, _ptr(sim),
                              _ptr(H) if H is not None else None)
    _check(rc, "orc_similarity")
    return (sim, H) if return_H else sim


def expert_counts(logits, kf):
    logits = _c(logits, np.float32); N, E = logits.shape
    cnt = np.empty(E, np.int32)
    _check(lib().orc_expert_counts(_ptr(logits), N, E, kf, _ptr(cnt)), "orc_expert_counts")
    return cnt


def theta(l, N, theta_min, theta_max, theta_single):
    return np.float32(lib().orc_theta(l, N, theta_min, theta_max, theta_single))


def group(sim, count, theta):
    sim = _c(sim, np.float32); count = _c(count, np.int32); E = sim.shape[0]
    g = np.empty(E, np.int32); K = ctypes.c_int32(0); dom = np.empty(E, np.int32)
    _check(lib().orc_group(_ptr(sim), _ptr(count), E, float(theta), _ptr(g), ctypes.byref(K),
                           _ptr(dom)), "orc_group")
    return g, int(K.value), dom[:K.value].copy()


def importance(sim, count, group, alpha_f=0.5, alpha_r=0.5):
    sim = _c(sim, np.float32); count = _c(count, np.int32); group = _c(group, np.int32)
    E = sim.shape[0]
    out = np.empty(E, np.float64)
    _check(lib().orc_importance(_ptr(sim), _ptr(count), _ptr(group), E, alpha_f, alpha_r, _ptr(out)),
           "orc_importance")
    return out


def place(group, importance, p, C, lambda1=0.5, lambda2=0.5):
    """group/importance/p: [L,E]; C: [M]. Returns (placement [L,M,E] u8, used [M], status)."""
    group = _c(group, np.int32); importance = _c(importance, np.float64)
    p = _c(p, np.float64); C = _c(C, np.float64)
    L, E = group.shape; M = C.shape[0]
    x = np.empty((L, M, E), np.uint8); used = np.empty(M, np.float64)
    rc = lib().orc_place(_ptr(group), _ptr(importance), _ptr(p), L, E, M, _ptr(C), lambda1, lambda2,
                         _ptr(x), _ptr(used))
    if rc not in (OK, CAPACITY):
        _check(rc, "orc_place")
    return x, used, rc


def replicate(group, importance, p, C, pi, placement, used):
    """Redundant deployment (Eqs. 32-35) after the mandatory placement.
    group/importance/p: [L,E]; C, pi, used: [M]; placement [L,M,E].
    Returns (placement, used, replicas [M]) as new arrays."""
    group = _c(group, np.int32); importance = _c(importance, np.float64)
    p = _c(p, np.float64); C = _c(C, np.float64); pi = _c(pi, np.float64)
    x = np.array(placement, dtype=np.uint8, copy=True, order="C")
    b = np.array(used, dtype=np.float64, copy=True, order="C")
    L, E = group.shape; M = C.shape[0]
    assert x.shape == (L, M, E) and b.shape == (M,) and pi.shape == (M,)
    reps = np.empty(M, np.int32)
    _check(lib().orc_replicate(_ptr(group), _ptr(importance), _ptr(p), L, E, M, _ptr(C), _ptr(pi),
                               _ptr(x), _ptr(b), _ptr(reps)), "orc_replicate")
    return x, b, reps


class _OrcTab(ctypes.Structure):
    _fields_ = [("Qtab", ctypes.c_void_p), ("Cq", ctypes.c_void_p), ("subst", ctypes.c_void_p),
                ("A", ctypes.c_void_p), ("pmask", ctypes.c_void_p)]


def phi(h, tabs, P, a, m, kx, qacc):
    """Eq. 42's cost-to-go Phi^(h) of orc_phi: tabs[0] is the current layer's
    Tables (not read), tabs[1..h] the next layers'; P [h, E, E] the transition
    matrices from the current layer on. Returns the fp32 value as a float."""
    t0 = tabs[0]
    arr = (_OrcTab * len(tabs))(*[_OrcTab(t.Qtab.ctypes.data, t.Cq.ctypes.data, t.subst.ctypes.data,
                                          t.A.ctypes.data, t.pmask.ctypes.data) for t in tabs])
    P = _c(P, np.float32)
    fn = lib().orc_phi
    fn.restype = ctypes.c_float
    fn.argtypes = [_I, ctypes.c_void_p, _P, _I, _I, _I, _I, _I, ctypes.c_float, ctypes.c_float]
    return float(fn(int(h), ctypes.cast(arr, ctypes.c_void_p), _ptr(P), t0.E, t0.M, int(a), int(m),
                    int(kx), ctypes.c_float(qacc), ctypes.c_float(t0.qbar)))


def trajectory_cost(target, chosen, server, home, F, B, tau, z, c, Qtab):
    """Edge delay / substitution loss / transfers of L layers' selection records
    (Eqs. 13-20). target/chosen/server: [L, T, k]; home [T]; Qtab [L, E, E].
    Returns (delay [T] f64, loss [T] f64, moves [T] i32)."""
    target = _c(target, np.int32); chosen = _c(chosen, np.int32); server = _c(server, np.uint8)
    home = _c(home, np.uint8); F = _c(F, np.float64); B = _c(B, np.float64)
    tau = _c(tau, np.float64); Qtab = _c(Qtab, np.float32)
    L, T, k = target.shape; E = Qtab.shape[-1]; M = F.shape[0]
    assert Qtab.shape == (L, E, E)
    d = np.empty(T, np.float64); q = np.empty(T, np.float64); n = np.empty(T, np.int32)
    _check(lib().orc_trajectory_cost(_ptr(target), _ptr(chosen), _ptr(server), _ptr(home), L, T, k,
                                     E, M, _ptr(F), _ptr(B), _ptr(tau), float(z), float(c),
                                     _ptr(Qtab), _ptr(d), _ptr(q), _ptr(n)), "orc_trajectory_cost")
    return d, q, n


def utility(delay, delay_ref, loss, qmax, omega_T, omega_Q, kappa):
    """Eq. 23 and Eq. 45: returns (U, Tbar, Qbar, omega_T', omega_Q')."""
    delay = _c(delay, np.float64); delay_ref = _c(delay_ref, np.float64); loss = _c(loss, np.float64)
    out = np.empty(5, np.float64)
    _check(lib().orc_utility(_ptr(delay), _ptr(delay_ref), _ptr(loss), delay.shape[0], float(qmax),
                             float(omega_T), float(omega_Q), float(kappa), _ptr(out)), "orc_utility")
    return tuple(float(v) for v in out)


def coverage(placement_l, group_l, K):
    placement_l = _c(placement_l, np.uint8); group_l = _c(group_l, np.int32)
    M, E = placement_l.shape
    cov = np.empty((M, K), np.uint8)
    _check(lib().orc_coverage(_ptr(placement_l), _ptr(group_l), E, M, K, _ptr(cov)), "orc_coverage")
    return cov


def transitions(logits, kf):
    """logits [N, L, E] f32 -> (counts [L-1, E, E] i32, P [L-1, E, E] f32), Eq. 41."""
    logits = _c(logits, np.float32)
    N, L, E = logits.shape
    cnt = np.empty((L - 1, E, E), np.int32); P = np.empty((L - 1, E, E), np.float32)
    _check(lib().orc_transitions(_ptr(logits), N, L, E, kf, _ptr(cnt), _ptr(P)), "orc_transitions")
    return cnt, P


def select_lookahead(idx, tabs, P, home, loc, qhat):
    """Alg. 2 with horizon H = len(tabs) (Eqs. 42-43); tabs[0] is the current layer's
    Tables, tabs[1:] the next layers'; P [H-1, E, E] the transition matrices."""
    idx = _c(idx, np.int32); T, k = idx.shape
    H = len(tabs); t0 = tabs[0]
    P = _c(P, np.float32).reshape(-1)
    if H > 1:
        assert P.size == (H - 1) * t0.E * t0.E
    else:
        P = np.zeros(1, np.float32)
    arr = lambda name, ct: (ct * max(H - 1, 1))(*[getattr(t, name).ctypes.data_as(ctypes.c_void_p)
                                                 for t in tabs[1:]] or [None])
    keep = [t for t in tabs]
    nQ, nC, nS, nA, nM = (arr(n, ctypes.c_void_p) for n in ("Qtab", "Cq", "subst", "A", "pmask"))
    home = _c(home, np.uint8); loc = _c(loc, np.uint8).copy(); qhat = _c(qhat, np.float32).copy()
    chosen = np.empty((T, k), np.int32); server = np.empty((T, k), np.uint8)
    kind = np.empty((T, k), np.uint8)
    rc = lib().orc_select_lookahead(_ptr(idx), T, t0.E, k, t0.M, H, _ptr(t0.Qtab), _ptr(t0.Cq),
                                    _ptr(t0.subst), _ptr(t0.A), _ptr(t0.pmask), nQ, nC, nS, nA, nM,
                                    _ptr(P), float(t0.qbar), _ptr(home), _ptr(loc), _ptr(qhat),
                                    _ptr(chosen), _ptr(server), _ptr(kind))
    del keep
    _check(rc, "orc_select_lookahead")
    return chosen, server, kind, loc, qhat
