"""The C ABI's argument checks, on the host without a GPU: a null pointer is
ORDERMOE_ERR_INVALID_ARG, a shape outside a call's stated limits (E <= 64
experts, M <= 32 servers, k <= 8 slots, the per-call multiples of d) is
ORDERMOE_ERR_UNSUPPORTED_SHAPE, both found before anything is enqueued, and
ordermoe_last_error() names the call, per thread. Only null device pointers
are passed, so no call can reach a kernel with an address it may not use."""
import threading

import pytest

from paper_2607_17154_gb300 import binding as B

N = None
# valid scalar arguments of each entry point, every pointer null; the prefix its
# messages start with
VALID = {
    "ordermoe_route_select": ([N, N, N, 16, 8, 64, 2, 1, N, 0] + [N] * 11, "route_select:"),
    "ordermoe_route_select_lookahead": ([N, N, N, 16, 8, 64, 2, 1, N, 0, 1] + [N] * 12,
                                        "route_select"),
    "ordermoe_dispatch": ([N, N, 16, 2, 8, 64, N, N, N, N, N, 0, N], "dispatch:"),
    "ordermoe_expert_ffn": ([N, N, 32, N, N, N, 8, 256, 512, N, N, N], "expert_ffn:"),
    "ordermoe_combine": ([N, N, N, 16, 2, 64, N, N], "combine:"),
    "ordermoe_rmsnorm": ([N, 16, 64, 1e-5, N, N], "rmsnorm:"),
    "ordermoe_similarity": ([N, N, 2, 8, 64, 1024, 2, N, N, N, 0, N], "similarity:"),
    "ordermoe_expert_counts": ([N, 100, 8, 2, N, N], "expert_counts:"),
    "ordermoe_transitions": ([N, 100, 2, 8, 2, N, N, N], "transitions:"),
    "ordermoe_build_tables": ([N, N, N, 8, 4, 0.5, 0.5, N, N, N, 1.0, 1.0, 1.0, 1.0, N, 0, N],
                              "build_tables:"),
    "ordermoe_place": ([N, N, 2, 8, 4, 0.5, 0.9, 0.5, 0.5, 0.5, 0.5, 0.5] + [N] * 10 + [0, N],
                       "place:"),
    "ordermoe_replicate": ([N, N, N, N, N, 2, 8, 4, N, N, N, N], "replicate:"),
    "ordermoe_coverage": ([N, N, 2, 8, 4, N, N, N], "coverage:"),
    "ordermoe_plan": ([N, N, 2, 8, 64, 1024, 2, 4, 0.5, 0.9, 0.5, 0.5, 0.5, 0.5, 0.5] + [N] * 16
                      + [0, N], "similarity:"),
}

# (entry, argument position, a value outside the stated limits)
SHAPES = [
    ("ordermoe_route_select", 4, 65), ("ordermoe_route_select", 6, 9),
    ("ordermoe_route_select", 6, 0), ("ordermoe_route_select_lookahead", 4, 65),
    ("ordermoe_route_select_lookahead", 10, 5), ("ordermoe_route_select_lookahead", 10, 0),
    ("ordermoe_dispatch", 4, 65), ("ordermoe_dispatch", 3, 0), ("ordermoe_dispatch", 3, 9),
    ("ordermoe_dispatch", 5, 12),
    ("ordermoe_expert_ffn", 6, 65), ("ordermoe_expert_ffn", 7, 128), ("ordermoe_expert_ffn", 8, 64),
    ("ordermoe_combine", 4, 0), ("ordermoe_combine", 4, 9), ("ordermoe_combine", 5, 12),
    ("ordermoe_rmsnorm", 2, 63),
    ("ordermoe_similarity", 3, 65), ("ordermoe_similarity", 4, 100), ("ordermoe_similarity", 6, 9),
    ("ordermoe_similarity", 2, 0), ("ordermoe_similarity", 5, 0),
    ("ordermoe_expert_counts", 2, 65), ("ordermoe_expert_counts", 3, 9),
    ("ordermoe_expert_counts", 3, 0),
    ("ordermoe_transitions", 3, 65), ("ordermoe_transitions", 4, 9), ("ordermoe_transitions", 2, 1),
    ("ordermoe_place", 3, 65), ("ordermoe_place", 4, 33), ("ordermoe_place", 4, 0),
    ("ordermoe_place", 2, 0),
    ("ordermoe_replicate", 6, 65), ("ordermoe_replicate", 7, 33), ("ordermoe_replicate", 5, 0),
    ("ordermoe_coverage", 3, 65), ("ordermoe_coverage", 4, 33), ("ordermoe_coverage", 2, 0),
    ("ordermoe_plan", 3, 65), ("ordermoe_plan", 4, 100),
]

# (entry, argument position) of a token or row count set to -1
NEGATIVE = [("ordermoe_route_select", 3), ("ordermoe_dispatch", 2), ("ordermoe_expert_ffn", 2),
            ("ordermoe_combine", 3), ("ordermoe_rmsnorm", 1)]


def run(name, args):
    L = B.lib()
    rc = getattr(L, name)(*args)
    msg = L.ordermoe_last_error()
    return rc, (msg.decode() if msg else "")


@pytest.mark.parametrize("name", sorted(VALID))
def test_null_pointers_are_invalid_arguments(name):
    args, prefix = VALID[name]
    rc, msg = run(name, args)
    assert rc == B.ERR_INVALID_ARG, (rc, msg)
    assert msg.startswith(prefix) and ("null" in msg or "pointer" in msg or "need P" in msg), msg


@pytest.mark.parametrize("name,pos,bad", SHAPES)
def test_shapes_outside_the_limits_are_unsupported(name, pos, bad):
    args, prefix = VALID[name]
    args = list(args)
    args[pos] = bad
    rc, msg = run(name, args)
    assert rc == B.ERR_UNSUPPORTED_SHAPE, (rc, msg)
    assert msg.startswith(prefix) and ("need" in msg or "must" in msg), msg


@pytest.mark.parametrize("name,pos", NEGATIVE)
def test_negative_counts_are_rejected(name, pos):
    args, prefix = VALID[name]
    args = list(args)
    args[pos] = -1
    rc, msg = run(name, args)
    assert rc in (B.ERR_INVALID_ARG, B.ERR_UNSUPPORTED_SHAPE), (rc, msg)
    assert msg.startswith(prefix), msg


def test_last_error_is_per_thread():
    """Two threads fail different calls at the same time; each reads its own
    message."""
    barrier = threading.Barrier(2)
    seen = {}

    def worker(tag, name, pos, bad):
        args = list(VALID[name][0])
        args[pos] = bad
        for _ in range(200):
            barrier.wait()
            rc, msg = run(name, args)
            barrier.wait()
            msg2 = B.lib().ordermoe_last_error().decode()
            seen.setdefault(tag, set()).add((rc, msg2))

    a = threading.Thread(target=worker, args=("a", "ordermoe_place", 4, 33))
    b = threading.Thread(target=worker, args=("b", "ordermoe_combine", 4, 9))
    a.start(); b.start(); a.join(); b.join()
    assert all(m.startswith("place:") for _, m in seen["a"]), seen["a"]
    assert all(m.startswith("combine:") for _, m in seen["b"]), seen["b"]
