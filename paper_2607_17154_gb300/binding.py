"""ctypes binding of libordermoe.so: one Python function per C-ABI entry point,
with the same names. Arguments are torch tensors on the current CUDA device;
the binding only checks dtypes/devices and passes pointers, sizes and the
current stream. Every step of the path runs in the library's kernels; there
is no fallback: if the library is missing the call raises.
"""
import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libordermoe.so")

OK = 0
ERR_INVALID_ARG, ERR_UNSUPPORTED_SHAPE, ERR_CAPACITY, ERR_CUDA, ERR_DEVICE_CHECK = 1, 2, 3, 4, 5
DEV_OK, DEV_NAN_LOGIT, DEV_BAD_INDEX, DEV_NO_CANDIDATE, DEV_WAIT_TIMEOUT, DEV_BAD_VALUE = 0, 1, 2, 3, 4, 5

_lib = None
_P = ctypes.c_void_p
_I = ctypes.c_int
_F = ctypes.c_float
_D = ctypes.c_double
_SZ = ctypes.c_size_t
_U64 = ctypes.c_uint64
_I64 = ctypes.c_int64

_SIGNATURES = {
    "ordermoe_version": ([], _I),
    "ordermoe_last_error": ([], ctypes.c_char_p),
    "ordermoe_device_error": ([_P, _P], _I),
    "ordermoe_set_wait_limit_ns": ([_U64], _I),
    "ordermoe_selftest_wait_timeout": ([_U64, _P], _I),
    "ordermoe_tables_bytes": ([_I, _I], _SZ),
    "ordermoe_build_tables": ([_P, _P, _P, _I, _I, _F, _F, _P, _P, _P, _D, _D, _D, _D, _P, _SZ, _P], _I),
    "ordermoe_route_select": ([_P, _P, _P, _I, _I, _I, _I, _I, _P, _SZ, _P, _P, _P, _P, _P, _P, _P,
                               _P, _P, _P, _P], _I),
    "ordermoe_dispatch_workspace_bytes": ([_I, _I, _I], _SZ),
    "ordermoe_dispatch": ([_P, _P, _I, _I, _I, _I, _P, _P, _P, _P, _P, _SZ, _P], _I),
    "ordermoe_expert_ffn": ([_P, _P, _I, _P, _P, _P, _I, _I, _I, _P, _P, _P], _I),
    "ordermoe_combine": ([_P, _P, _P, _I, _I, _I, _P, _P], _I),
    "ordermoe_similarity_workspace_bytes": ([_I, _I, _I64], _SZ),
    "ordermoe_similarity": ([_P, _P, _I, _I, _I, _I64, _I, _P, _P, _P, _SZ, _P], _I),
    "ordermoe_similarity_no_logits": ([_P, _P, _I, _I, _I, _I64, _I, _P, _P, _P, _SZ, _P], _I),
    "ordermoe_expert_counts": ([_P, _I64, _I, _I, _P, _P], _I),
    "ordermoe_place": ([_P, _P, _I, _I, _I, _D, _D, _D, _D, _D, _D, _D, _P, _P, _P, _P, _P, _P,
                        _P, _P, _P, _P, _SZ, _P], _I),
    "ordermoe_replicate": ([_P, _P, _P, _P, _P, _I, _I, _I, _P, _P, _P, _P], _I),
    "ordermoe_coverage": ([_P, _P, _I, _I, _I, _P, _P, _P], _I),
    "ordermoe_trajectory_cost": ([_P, _P, _P, _P, _I, _I, _I, _I, _P, _SZ, _I, _P, _P, _P, _D, _D,
                                  _P, _P, _P, _P], _I),
    "ordermoe_utility": ([_P, _P, _P, _I, _D, _D, _D, _D, _P, _P], _I),
    "ordermoe_selftest_div_rn": ([_P, _P, _P, _I64, _P], _I),
    "ordermoe_layer_batches_scratch_bytes": ([_I, _I, _I, _I, _I], _SZ),
    "ordermoe_layer_forward_batches": ([_P, _I, _I, _P, _P, _P, _P, _P], _I),
    "ordermoe_place_workspace_bytes": ([_I, _I], _SZ),
    "ordermoe_expert_gate_up": ([_P, _P, _I, _P, _P, _I, _I, _I, _P, _P], _I),
    "ordermoe_expert_down": ([_P, _P, _I, _P, _I, _I, _I, _P, _P], _I),
    "ordermoe_layer_scratch_bytes": ([_I, _I, _I, _I, _I], _SZ),
    "ordermoe_layer_forward": ([_P, _I, _P, _P, _P, _P, _P, _P, _I, _P], _I),
    "ordermoe_dispatch_noalloc": ([_P, _P, _I, _I, _I, _I, _P, _P, _P, _P, _P], _I),
    "ordermoe_transitions": ([_P, _I64, _I, _I, _I, _P, _P, _P], _I),
    "ordermoe_plan_workspace_bytes": ([_I, _I, _I64], _SZ),
    "ordermoe_plan": ([_P, _P, _I, _I, _I, _I64, _I, _I, _D, _D, _D, _D, _D, _D, _D, _P, _P, _P,
                       _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _SZ, _P], _I),
    "ordermoe_route_select_lookahead": ([_P, _P, _P, _I, _I, _I, _I, _I, _P, _SZ, _I, _P, _P, _P,
                                         _P, _P, _P, _P, _P, _P, _P, _P, _P], _I),
    "ordermoe_rmsnorm": ([_P, _I, _I, _F, _P, _P], _I),
    "ordermoe_combine_residual_norm": ([_P, _P, _P, _P, _I, _I, _I, _F, _P, _P, _P], _I),
    "ordermoe_layer_forward_residual": ([_P, _I, _P, _P, _P, _P, _P, _F, _P, _P, _P, _P, _P], _I),
    "ordermoe_transitions_strided": ([_P, _I64, _I, _I, _I, _I64, _I64, _P, _P, _P], _I),
}

# RMSNorm epsilon of the residual map between stacked layers
NORM_EPS = 1e-6


class LayerDesc(ctypes.Structure):
    """Mirror of ordermoe_layer_desc."""
    _fields_ = [("T_max", _I), ("E", _I), ("d", _I), ("dff", _I), ("k", _I), ("renorm", _I),
                ("W_r", _P), ("W1", _P), ("W3", _P), ("W2", _P), ("tables", _P),
                ("tables_bytes", _SZ), ("scratch", _P), ("scratch_bytes", _SZ),
                ("lookahead_H", _I), ("tables_stride", _SZ), ("P", _P)]


class OrderMoEError(RuntimeError):
    def __init__(self, name, code, msg):
        super().__init__("%s failed with status %d: %s" % (name, code, msg))
        self.code = code


def lib():
    """Load libordermoe.so (built in-tree by build.py / __graft_entry__.build())."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libordermoe.so is not built (%s); run __graft_entry__.build()"
                               % LIB_PATH)
        L = ctypes.CDLL(LIB_PATH)
        for name, (args, res) in _SIGNATURES.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = res
        _lib = L
    return _lib


def _check(name, rc):
    if rc != OK:
        msg = lib().ordermoe_last_error()
        raise OrderMoEError(name, rc, msg.decode() if msg else "")


def _ptr(t):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        raise TypeError("expected a torch.Tensor")
    if not t.is_cuda:
        raise ValueError("tensor must be on a CUDA device")
    if not t.is_contiguous():
        raise ValueError("tensor must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _dt(t, dtype, name):
    if t is not None and t.dtype != dtype:
        raise TypeError("%s must be %s, got %s" % (name, dtype, t.dtype))


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


# ------------------------------------------------------------------ entry points

def ordermoe_version():
    return lib().ordermoe_version()


def ordermoe_device_error():
    """Synchronises; returns (code, detail) of the device error word and clears it."""
    code = ctypes.c_int(0); detail = ctypes.c_int(0)
    lib().ordermoe_device_error(ctypes.byref(code), ctypes.byref(detail))
    return code.value, detail.value


def ordermoe_set_wait_limit_ns(limit_ns):
    _check("ordermoe_set_wait_limit_ns", lib().ordermoe_set_wait_limit_ns(int(limit_ns)))


def ordermoe_selftest_wait_timeout(limit_ns, stream=None):
    _check("ordermoe_selftest_wait_timeout",
           lib().ordermoe_selftest_wait_timeout(int(limit_ns), _stream(stream)))


def ordermoe_tables_bytes(E, M):
    return int(lib().ordermoe_tables_bytes(E, M))


def ordermoe_build_tables(sim, group, placement, theta, qbar, F, B, tau, z, c, omega_T, omega_Q,
                          tables, stream=None):
    _dt(sim, torch.float32, "sim"); _dt(group, torch.int32, "group")
    _dt(placement, torch.uint8, "placement"); _dt(tables, torch.uint8, "tables")
    for n, t in (("F", F), ("B", B), ("tau", tau)):
        _dt(t, torch.float64, n)
    E = sim.shape[0]; M = placement.shape[0]
    rc = lib().ordermoe_build_tables(_ptr(sim), _ptr(group), _ptr(placement), E, M, float(theta),
                                     float(qbar), _ptr(F), _ptr(B), _ptr(tau), float(z), float(c),
                                     float(omega_T), float(omega_Q), _ptr(tables), tables.numel(),
                                     _stream(stream))
    _check("ordermoe_build_tables", rc)


def ordermoe_route_select(X, W_r, logits_in, T, E, d, k, renorm, tables, home, loc, qhat,
                          logits_out, topk_idx, topk_w, chosen_expert, chosen_server, kind,
                          counters=None, stream=None):
    _dt(X, torch.bfloat16, "X"); _dt(W_r, torch.bfloat16, "W_r"); _dt(logits_in, torch.float32, "logits_in")
    _dt(home, torch.uint8, "home"); _dt(loc, torch.uint8, "loc"); _dt(qhat, torch.float32, "qhat")
    _dt(topk_idx, torch.int32, "topk_idx"); _dt(topk_w, torch.float32, "topk_w")
    _dt(chosen_expert, torch.int32, "chosen_expert"); _dt(chosen_server, torch.uint8, "chosen_server")
    _dt(kind, torch.uint8, "kind"); _dt(counters, torch.int32, "counters")
    rc = lib().ordermoe_route_select(_ptr(X), _ptr(W_r), _ptr(logits_in), T, E, d, k, int(renorm),
                                     _ptr(tables), tables.numel(), _ptr(home), _ptr(loc), _ptr(qhat),
                                     _ptr(logits_out), _ptr(topk_idx), _ptr(topk_w),
                                     _ptr(chosen_expert), _ptr(chosen_server), _ptr(kind),
                                     _ptr(counters), _stream(stream))
    _check("ordermoe_route_select", rc)


def ordermoe_dispatch_workspace_bytes(T, k, E):
    return int(lib().ordermoe_dispatch_workspace_bytes(T, k, E))


def ordermoe_dispatch(chosen_expert, X, T, k, E, d, offsets, row_token, row_of, X_perm, workspace,
                      stream=None):
    _dt(chosen_expert, torch.int32, "chosen_expert"); _dt(X, torch.bfloat16, "X")
    _dt(offsets, torch.int32, "offsets"); _dt(row_token, torch.int32, "row_token")
    _dt(row_of, torch.int32, "row_of"); _dt(X_perm, torch.bfloat16, "X_perm")
    rc = lib().ordermoe_dispatch(_ptr(chosen_expert), _ptr(X), T, k, E, d, _ptr(offsets),
                                 _ptr(row_token), _ptr(row_of), _ptr(X_perm), _ptr(workspace),
                                 workspace.numel() * workspace.element_size(), _stream(stream))
    _check("ordermoe_dispatch", rc)


def ordermoe_expert_ffn(X_perm, offsets, R, W1, W3, W2, E, d, dff, H, Y_perm, stream=None):
    for n, t in (("X_perm", X_perm), ("W1", W1), ("W3", W3), ("W2", W2), ("H", H), ("Y_perm", Y_perm)):
        _dt(t, torch.bfloat16, n)
    _dt(offsets, torch.int32, "offsets")
    rc = lib().ordermoe_expert_ffn(_ptr(X_perm), _ptr(offsets), R, _ptr(W1), _ptr(W3), _ptr(W2),
                                   E, d, dff, _ptr(H), _ptr(Y_perm), _stream(stream))
    _check("ordermoe_expert_ffn", rc)


def ordermoe_combine(Y_perm, row_of, topk_w, T, k, d, y, stream=None):
    _dt(Y_perm, torch.bfloat16, "Y_perm"); _dt(row_of, torch.int32, "row_of")
    _dt(topk_w, torch.float32, "topk_w"); _dt(y, torch.bfloat16, "y")
    rc = lib().ordermoe_combine(_ptr(Y_perm), _ptr(row_of), _ptr(topk_w), T, k, d, _ptr(y),
                                _stream(stream))
    _check("ordermoe_combine", rc)


def ordermoe_similarity_workspace_bytes(L, E, N):
    return int(lib().ordermoe_similarity_workspace_bytes(L, E, N))


def ordermoe_similarity(W_r, X_cal, L, E, d, N, k_freq, sim, counts, workspace, stream=None):
    _dt(W_r, torch.bfloat16, "W_r"); _dt(X_cal, torch.bfloat16, "X_cal")
    _dt(sim, torch.float32, "sim"); _dt(counts, torch.int32, "counts")
    rc = lib().ordermoe_similarity(_ptr(W_r), _ptr(X_cal), L, E, d, N, k_freq, _ptr(sim),
                                   _ptr(counts), _ptr(workspace),
                                   workspace.numel() * workspace.element_size(), _stream(stream))
    _check("ordermoe_similarity", rc)


def ordermoe_similarity_no_logits(W_r, X_cal, L, E, d, N, k_freq, sim, counts, workspace,
                                  stream=None):
    _dt(W_r, torch.bfloat16, "W_r"); _dt(X_cal, torch.bfloat16, "X_cal")
    _dt(sim, torch.float32, "sim"); _dt(counts, torch.int32, "counts")
    rc = lib().ordermoe_similarity_no_logits(_ptr(W_r), _ptr(X_cal), L, E, d, N, k_freq,
                                             _ptr(sim), _ptr(counts), _ptr(workspace),
                                             workspace.numel() * workspace.element_size(),
                                             _stream(stream))
    _check("ordermoe_similarity_no_logits", rc)


def ordermoe_expert_counts(logits, N, E, k_freq, counts, stream=None):
    _dt(logits, torch.float32, "logits"); _dt(counts, torch.int32, "counts")
    _check("ordermoe_expert_counts",
           lib().ordermoe_expert_counts(_ptr(logits), N, E, k_freq, _ptr(counts), _stream(stream)))


def ordermoe_place_workspace_bytes(L, E):
    return int(lib().ordermoe_place_workspace_bytes(L, E))


def ordermoe_place(sim, counts, L, E, M, theta_min, theta_max, theta_single, alpha_f, alpha_r,
                   lambda1, lambda2, p, C, group, n_groups, theta, importance, placement, used,
                   status, workspace=None, stream=None):
    """importance: [L, E] f64 output or None. workspace: device scratch of
    ordermoe_place_workspace_bytes(L, E) bytes; allocated here with torch when
    not given."""
    if workspace is None:
        workspace = torch.empty(ordermoe_place_workspace_bytes(L, E), dtype=torch.uint8,
                                device=sim.device)
    _dt(sim, torch.float32, "sim"); _dt(counts, torch.int32, "counts")
    _dt(p, torch.float64, "p"); _dt(C, torch.float64, "C"); _dt(group, torch.int32, "group")
    _dt(n_groups, torch.int32, "n_groups"); _dt(theta, torch.float32, "theta")
    _dt(placement, torch.uint8, "placement"); _dt(used, torch.float64, "used")
    _dt(status, torch.int32, "status"); _dt(importance, torch.float64, "importance")
    rc = lib().ordermoe_place(_ptr(sim), _ptr(counts), L, E, M, float(theta_min), float(theta_max),
                              float(theta_single), float(alpha_f), float(alpha_r), float(lambda1),
                              float(lambda2), _ptr(p), _ptr(C), _ptr(group), _ptr(n_groups),
                              _ptr(theta), _ptr(importance), _ptr(placement), _ptr(used), _ptr(status),
                              _ptr(workspace), workspace.numel() * workspace.element_size(),
                              _stream(stream))
    _check("ordermoe_place", rc)


def ordermoe_replicate(group, importance, p, C, pi, L, E, M, placement, used, replicas, stream=None):
    """Redundant deployment (Eqs. 32-35); placement and used are updated in place."""
    _dt(group, torch.int32, "group"); _dt(importance, torch.float64, "importance")
    _dt(p, torch.float64, "p"); _dt(C, torch.float64, "C"); _dt(pi, torch.float64, "pi")
    _dt(placement, torch.uint8, "placement"); _dt(used, torch.float64, "used")
    _dt(replicas, torch.int32, "replicas")
    _check("ordermoe_replicate", lib().ordermoe_replicate(
        _ptr(group), _ptr(importance), _ptr(p), _ptr(C), _ptr(pi), L, E, M, _ptr(placement),
        _ptr(used), _ptr(replicas), _stream(stream)))


def ordermoe_coverage(group, placement, L, E, M, cover=None, covered=None, stream=None):
    """Local group coverage (Eq. 32): cover [L, M, E] u8 and covered [L] i32 (either may be None)."""
    _dt(group, torch.int32, "group"); _dt(placement, torch.uint8, "placement")
    _dt(cover, torch.uint8, "cover"); _dt(covered, torch.int32, "covered")
    _check("ordermoe_coverage", lib().ordermoe_coverage(_ptr(group), _ptr(placement), L, E, M,
                                                        _ptr(cover), _ptr(covered), _stream(stream)))


def ordermoe_plan_workspace_bytes(L, E, N):
    return int(lib().ordermoe_plan_workspace_bytes(L, E, N))


def ordermoe_plan(W_r, X_cal, L, E, d, N, k_freq, M, theta_min, theta_max, theta_single, alpha_f,
                  alpha_r, lambda1, lambda2, p, C, pi, sim, counts, group, n_groups, theta,
                  importance, placement, used, status, replicas, cover, covered, workspace,
                  stream=None):
    """The whole offline plan (similarity, grouping, placement, redundancy,
    coverage) in one call; workspace: ordermoe_plan_workspace_bytes(L, E, N) bytes."""
    _dt(W_r, torch.bfloat16, "W_r"); _dt(X_cal, torch.bfloat16, "X_cal")
    for n, v in (("p", p), ("C", C), ("pi", pi), ("importance", importance), ("used", used)):
        _dt(v, torch.float64, n)
    _dt(sim, torch.float32, "sim"); _dt(counts, torch.int32, "counts"); _dt(group, torch.int32, "group")
    _dt(n_groups, torch.int32, "n_groups"); _dt(theta, torch.float32, "theta")
    _dt(placement, torch.uint8, "placement"); _dt(status, torch.int32, "status")
    _dt(replicas, torch.int32, "replicas"); _dt(cover, torch.uint8, "cover")
    _dt(covered, torch.int32, "covered"); _dt(workspace, torch.uint8, "workspace")
    _check("ordermoe_plan", lib().ordermoe_plan(
        _ptr(W_r), _ptr(X_cal), L, E, d, N, k_freq, M, float(theta_min), float(theta_max),
        float(theta_single), float(alpha_f), float(alpha_r), float(lambda1), float(lambda2), _ptr(p),
        _ptr(C), _ptr(pi), _ptr(sim), _ptr(counts), _ptr(group), _ptr(n_groups), _ptr(theta),
        _ptr(importance), _ptr(placement), _ptr(used), _ptr(status), _ptr(replicas), _ptr(cover),
        _ptr(covered), _ptr(workspace), workspace.numel(), _stream(stream)))


def ordermoe_trajectory_cost(target, chosen_expert, chosen_server, home, L, T, k, E, tables,
                             tables_stride, M, F, B, tau, z, c, delay, loss, moves, stream=None):
    """Edge delay, substitution loss and transfers of L layers' records (Eqs. 13-20)."""
    _dt(target, torch.int32, "target"); _dt(chosen_expert, torch.int32, "chosen_expert")
    _dt(chosen_server, torch.uint8, "chosen_server"); _dt(home, torch.uint8, "home")
    for n, v in (("F", F), ("B", B), ("tau", tau), ("delay", delay), ("loss", loss)):
        _dt(v, torch.float64, n)
    _dt(moves, torch.int32, "moves")
    _check("ordermoe_trajectory_cost", lib().ordermoe_trajectory_cost(
        _ptr(target), _ptr(chosen_expert), _ptr(chosen_server), _ptr(home), L, T, k, E, _ptr(tables),
        int(tables_stride), M, _ptr(F), _ptr(B), _ptr(tau), float(z), float(c), _ptr(delay),
        _ptr(loss), _ptr(moves), _stream(stream)))


def ordermoe_utility(delay, delay_ref, loss, T, qmax, omega_T, omega_Q, kappa, out, stream=None):
    """Eq. 23 and Eq. 45 into out [5] f64: U, Tbar, Qbar, omega_T', omega_Q'."""
    for n, v in (("delay", delay), ("delay_ref", delay_ref), ("loss", loss), ("out", out)):
        _dt(v, torch.float64, n)
    _check("ordermoe_utility", lib().ordermoe_utility(
        _ptr(delay), _ptr(delay_ref), _ptr(loss), T, float(qmax), float(omega_T), float(omega_Q),
        float(kappa), _ptr(out), _stream(stream)))


def ordermoe_selftest_div_rn(a, b, out, stream=None):
    """out = a / b as the placement computes its load ratios (f64 device tensors)."""
    for n, v in (("a", a), ("b", b), ("out", out)):
        _dt(v, torch.float64, n)
    _check("ordermoe_selftest_div_rn", lib().ordermoe_selftest_div_rn(
        _ptr(a), _ptr(b), _ptr(out), a.numel(), _stream(stream)))


def ordermoe_expert_gate_up(X_perm, offsets, R, W1, W3, E, d, dff, H, stream=None):
    for n, t in (("X_perm", X_perm), ("W1", W1), ("W3", W3), ("H", H)):
        _dt(t, torch.bfloat16, n)
    _dt(offsets, torch.int32, "offsets")
    _check("ordermoe_expert_gate_up",
           lib().ordermoe_expert_gate_up(_ptr(X_perm), _ptr(offsets), R, _ptr(W1), _ptr(W3), E, d,
                                         dff, _ptr(H), _stream(stream)))


def ordermoe_expert_down(H, offsets, R, W2, E, d, dff, Y_perm, stream=None):
    for n, t in (("H", H), ("W2", W2), ("Y_perm", Y_perm)):
        _dt(t, torch.bfloat16, n)
    _dt(offsets, torch.int32, "offsets")
    _check("ordermoe_expert_down",
           lib().ordermoe_expert_down(_ptr(H), _ptr(offsets), R, _ptr(W2), E, d, dff, _ptr(Y_perm),
                                      _stream(stream)))


def ordermoe_layer_scratch_bytes(T_max, E, d, dff, k):
    return int(lib().ordermoe_layer_scratch_bytes(T_max, E, d, dff, k))


def make_layer_desc(T_max, W_r, W1, W3, W2, tables, k, scratch, renorm=1, lookahead_H=1,
                    tables_stride=0, P=None):
    """tables: this layer's tables (uint8 device tensor); with lookahead_H > 1 it
    must continue with the next layers' tables at tables_stride bytes."""
    E, dff, d = W1.shape
    for n, t in (("W_r", W_r), ("W1", W1), ("W3", W3), ("W2", W2)):
        _dt(t, torch.bfloat16, n)
    _dt(P, torch.float32, "P")
    desc = LayerDesc(T_max, E, d, dff, k, int(renorm), _ptr(W_r), _ptr(W1), _ptr(W3), _ptr(W2),
                     _ptr(tables), tables.numel(), _ptr(scratch),
                     scratch.numel() * scratch.element_size(), int(lookahead_H), int(tables_stride),
                     _ptr(P))
    desc._keep = (W_r, W1, W3, W2, tables, scratch, P)
    return desc


def _host_or_dev_ptr(t, host):
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensor must be contiguous")
    if host and t.is_cuda:
        raise ValueError("host_io=1 needs host tensors")
    if not host and not t.is_cuda:
        raise ValueError("host_io=0 needs CUDA tensors")
    return ctypes.c_void_p(t.data_ptr())


def ordermoe_layer_forward(desc, T, X, home, loc, qhat, y, counters=None, host_io=0, stream=None):
    h = bool(host_io)
    _dt(X, torch.bfloat16, "X"); _dt(y, torch.bfloat16, "y"); _dt(home, torch.uint8, "home")
    _dt(loc, torch.uint8, "loc"); _dt(qhat, torch.float32, "qhat")
    rc = lib().ordermoe_layer_forward(ctypes.byref(desc), T, _host_or_dev_ptr(X, h),
                                      _host_or_dev_ptr(home, h), _host_or_dev_ptr(loc, h),
                                      _host_or_dev_ptr(qhat, h), _host_or_dev_ptr(y, h),
                                      _ptr(counters), int(host_io), _stream(stream))
    _check("ordermoe_layer_forward", rc)


def ordermoe_rmsnorm(h, T, d, eps, x, stream=None):
    _dt(h, torch.bfloat16, "h"); _dt(x, torch.bfloat16, "x")
    _check("ordermoe_rmsnorm", lib().ordermoe_rmsnorm(_ptr(h), T, d, float(eps), _ptr(x),
                                                      _stream(stream)))


def ordermoe_combine_residual_norm(Y_perm, row_of, topk_w, h, T, k, d, eps, h_out, x_out,
                                   stream=None):
    _dt(Y_perm, torch.bfloat16, "Y_perm"); _dt(row_of, torch.int32, "row_of")
    _dt(topk_w, torch.float32, "topk_w")
    for n, t in (("h", h), ("h_out", h_out), ("x_out", x_out)):
        _dt(t, torch.bfloat16, n)
    rc = lib().ordermoe_combine_residual_norm(_ptr(Y_perm), _ptr(row_of), _ptr(topk_w), _ptr(h), T,
                                              k, d, float(eps), _ptr(h_out), _ptr(x_out),
                                              _stream(stream))
    _check("ordermoe_combine_residual_norm", rc)


def ordermoe_layer_forward_residual(desc, T, x, h, home, loc, qhat, eps, h_out, x_out,
                                    logits_out=None, counters=None, stream=None):
    for n, t in (("x", x), ("h", h), ("h_out", h_out), ("x_out", x_out)):
        _dt(t, torch.bfloat16, n)
    _dt(home, torch.uint8, "home"); _dt(loc, torch.uint8, "loc"); _dt(qhat, torch.float32, "qhat")
    _dt(logits_out, torch.float32, "logits_out")
    rc = lib().ordermoe_layer_forward_residual(ctypes.byref(desc), T, _ptr(x), _ptr(h), _ptr(home),
                                               _ptr(loc), _ptr(qhat), float(eps), _ptr(h_out),
                                               _ptr(x_out), _ptr(logits_out), _ptr(counters),
                                               _stream(stream))
    _check("ordermoe_layer_forward_residual", rc)


def ordermoe_layer_batches_scratch_bytes(T_max, E, d, dff, k):
    return int(lib().ordermoe_layer_batches_scratch_bytes(T_max, E, d, dff, k))


def ordermoe_layer_forward_batches(desc, nbatch, T, X, home, y, counters=None, stream=None):
    """X [nbatch, T, d] bf16, home [nbatch, T] u8, y [nbatch, T, d] bf16: pinned host tensors."""
    _dt(X, torch.bfloat16, "X"); _dt(y, torch.bfloat16, "y"); _dt(home, torch.uint8, "home")
    for n, t in (("X", X), ("home", home), ("y", y)):
        if t.is_cuda or not t.is_contiguous():
            raise ValueError("%s must be a contiguous host tensor" % n)
    rc = lib().ordermoe_layer_forward_batches(ctypes.byref(desc), int(nbatch), int(T),
                                              _host_or_dev_ptr(X, True), _host_or_dev_ptr(home, True),
                                              _host_or_dev_ptr(y, True), _ptr(counters), _stream(stream))
    _check("ordermoe_layer_forward_batches", rc)


def ordermoe_dispatch_noalloc(chosen_expert, X, T, k, E, d, offsets, row_token, row_of, X_perm,
                              stream=None):
    """ordermoe_dispatch without a workspace argument: for callers that cannot
    allocate device memory (the library keeps a fixed 256 KB scratch array)."""
    _dt(chosen_expert, torch.int32, "chosen_expert"); _dt(X, torch.bfloat16, "X")
    _dt(offsets, torch.int32, "offsets"); _dt(row_token, torch.int32, "row_token")
    _dt(row_of, torch.int32, "row_of"); _dt(X_perm, torch.bfloat16, "X_perm")
    rc = lib().ordermoe_dispatch_noalloc(_ptr(chosen_expert), _ptr(X), T, k, E, d, _ptr(offsets),
                                         _ptr(row_token), _ptr(row_of), _ptr(X_perm),
                                         _stream(stream))
    _check("ordermoe_dispatch_noalloc", rc)


def ordermoe_transitions(logits, N, L, E, k_freq, counts, P, stream=None):
    _dt(logits, torch.float32, "logits"); _dt(counts, torch.int32, "counts"); _dt(P, torch.float32, "P")
    _check("ordermoe_transitions",
           lib().ordermoe_transitions(_ptr(logits), N, L, E, k_freq, _ptr(counts), _ptr(P),
                                      _stream(stream)))


def ordermoe_transitions_strided(logits, N, L, E, k_freq, token_stride, layer_stride, counts, P,
                                 stream=None):
    _dt(logits, torch.float32, "logits"); _dt(counts, torch.int32, "counts"); _dt(P, torch.float32, "P")
    _check("ordermoe_transitions_strided",
           lib().ordermoe_transitions_strided(_ptr(logits), N, L, E, k_freq, int(token_stride),
                                              int(layer_stride), _ptr(counts), _ptr(P),
                                              _stream(stream)))


def ordermoe_route_select_lookahead(X, W_r, logits_in, T, E, d, k, renorm, tables, tables_stride, H,
                                    P, home, loc, qhat, logits_out, topk_idx, topk_w,
                                    chosen_expert, chosen_server, kind, counters=None, stream=None):
    """tables: a uint8 device tensor holding H (or more) consecutive layer tables,
    tables_stride bytes apart, starting with this layer's."""
    _dt(X, torch.bfloat16, "X"); _dt(W_r, torch.bfloat16, "W_r"); _dt(logits_in, torch.float32, "logits_in")
    _dt(P, torch.float32, "P")
    rc = lib().ordermoe_route_select_lookahead(
        _ptr(X), _ptr(W_r), _ptr(logits_in), T, E, d, k, int(renorm), _ptr(tables), int(tables_stride),
        int(H), _ptr(P), _ptr(home), _ptr(loc), _ptr(qhat), _ptr(logits_out), _ptr(topk_idx),
        _ptr(topk_w), _ptr(chosen_expert), _ptr(chosen_server), _ptr(kind), _ptr(counters),
        _stream(stream))
    _check("ordermoe_route_select_lookahead", rc)
