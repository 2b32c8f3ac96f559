"""The CUDA path reproduces the golden fixtures (expected values written by
the oracle alone): one layer's tables and selection, and the three-layer
placement with redundancy."""
import json
import os

import numpy as np
import pytest
import torch

from paper_2607_17154_gb300 import binding as B
from paper_2607_17154_gb300 import synth

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    B.lib()
    yield
    code, detail = B.ordermoe_device_error()
    assert code == 0, (code, detail)


def fixture(name):
    with open(os.path.join(GOLDEN, name + ".json")) as f:
        d = json.load(f)

    def dec(v):
        if isinstance(v, dict) and "hex" in v:
            return np.frombuffer(bytes.fromhex(v["hex"]), dtype=np.dtype(v["dtype"])).reshape(v["shape"])
        return v
    return {k: dec(v) for k, v in d["inputs"].items()}, {k: dec(v) for k, v in d["outputs"].items()}


def g(a, dt):
    return torch.as_tensor(np.array(a, copy=True)).to(device=DEV, dtype=dt)


def test_selection_fixture():
    inp, out = fixture("selection_one_layer")
    E = inp["sim"].shape[0]; M = inp["placement"].shape[0]; k = inp["k"]; T = inp["logits"].shape[0]
    tab = torch.zeros(B.ordermoe_tables_bytes(E, M), dtype=torch.uint8, device=DEV)
    B.ordermoe_build_tables(g(inp["sim"], torch.float32), g(inp["group"], torch.int32),
                            g(inp["placement"], torch.uint8), inp["theta"], inp["qbar"],
                            g(inp["F"], torch.float64), g(inp["B"], torch.float64),
                            g(inp["tau"], torch.float64), inp["z"], inp["c"], 0.5, 0.5, tab)
    raw = tab.cpu().numpy()
    off_q = 832
    Q = raw[off_q:off_q + 4 * E * E].view(np.float32).reshape(E, E)
    Cq = raw[off_q + 4 * E * E:off_q + 8 * E * E].view(np.float32).reshape(E, E)
    A = raw[off_q + 8 * E * E:off_q + 8 * E * E + 4 * M * M * M].view(np.float32)
    np.testing.assert_array_equal(Q, out["Qtab"])
    np.testing.assert_array_equal(Cq, out["Cq"])
    np.testing.assert_array_equal(A, np.asarray(out["A"]).reshape(-1))
    outs = [torch.empty(T, k, dtype=dt, device=DEV)
            for dt in (torch.int32, torch.float32, torch.int32, torch.uint8, torch.uint8)]
    loc = g(inp["loc"], torch.uint8); qhat = g(inp["qhat"], torch.float32)
    B.ordermoe_route_select(None, None, g(inp["logits"], torch.float32), T, E, 0, k, 1, tab,
                            g(inp["home"], torch.uint8), loc, qhat, None, *outs)
    for name, t in zip(("topk_idx", "chosen", "server", "kind"), (outs[0], outs[2], outs[3], outs[4])):
        np.testing.assert_array_equal(t.cpu().numpy(), out[name], err_msg=name)
    np.testing.assert_allclose(outs[1].cpu().numpy(), out["topk_w"], rtol=1e-5, atol=1e-7)
    np.testing.assert_array_equal(loc.cpu().numpy(), out["loc"])
    np.testing.assert_array_equal(qhat.cpu().numpy(), out["qhat"])


def test_plan_fixture():
    inp, out = fixture("plan_three_layers")
    L, E = out["group"].shape; M = inp["C"].shape[0]
    group = torch.empty(L, E, dtype=torch.int32, device=DEV)
    ng = torch.empty(L, dtype=torch.int32, device=DEV)
    theta = torch.empty(L, dtype=torch.float32, device=DEV)
    imp = torch.empty(L, E, dtype=torch.float64, device=DEV)
    x = torch.empty(L, M, E, dtype=torch.uint8, device=DEV)
    used = torch.empty(M, dtype=torch.float64, device=DEV)
    st = torch.empty(1, dtype=torch.int32, device=DEV)
    gp, gC = g(inp["p"], torch.float64), g(inp["C"], torch.float64)
    B.ordermoe_place(g(out["sim"], torch.float32), g(out["counts"], torch.int32), L, E, M, 0.5, 0.9,
                     0.5, 0.5, 0.5, 0.5, 0.5, gp, gC, group, ng, theta, imp, x, used, st)
    np.testing.assert_array_equal(group.cpu().numpy(), out["group"])
    np.testing.assert_array_equal(theta.cpu().numpy(), out["theta"].astype(np.float32))
    np.testing.assert_array_equal(imp.cpu().numpy(), out["importance"])
    np.testing.assert_array_equal(x.cpu().numpy(), out["placement"])
    np.testing.assert_array_equal(used.cpu().numpy(), out["used"])
    assert st.item() == out["status"]
    reps = torch.empty(M, dtype=torch.int32, device=DEV)
    B.ordermoe_replicate(group, imp, gp, gC, g(inp["pi"], torch.float64), L, E, M, x, used, reps)
    np.testing.assert_array_equal(x.cpu().numpy(), out["placement_redundant"])
    np.testing.assert_array_equal(used.cpu().numpy(), out["used_redundant"])
    np.testing.assert_array_equal(reps.cpu().numpy(), out["replicas"])
