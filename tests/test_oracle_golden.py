"""The oracle still reproduces the golden fixtures of tests/golden exactly
(inputs regenerated from their seeds, every output compared byte for byte).
The fixtures were written by tests/golden/make_golden.py from the oracle alone;
a deliberate change to the oracle's arithmetic regenerates them."""
import importlib.util
import json
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def load_maker():
    spec = importlib.util.spec_from_file_location("make_golden", os.path.join(GOLDEN, "make_golden.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def decode(v):
    if isinstance(v, dict) and "hex" in v:
        return np.frombuffer(bytes.fromhex(v["hex"]), dtype=np.dtype(v["dtype"])).reshape(v["shape"])
    return v


@pytest.mark.parametrize("name", ["selection_one_layer", "plan_three_layers", "lookahead_and_edge_cost"])
def test_oracle_reproduces_golden_fixture(name):
    maker = load_maker()
    with open(os.path.join(GOLDEN, name + ".json")) as f:
        stored = json.load(f)
    assert stored["cite"]
    case = maker.CASES[name]()
    for part in ("inputs", "outputs"):
        assert set(case[part]) == set(stored[part]), part
        for key, val in case[part].items():
            want = decode(stored[part][key])
            got = maker.encode(val)
            got = decode(got)
            if isinstance(want, np.ndarray):
                assert got.dtype == want.dtype and got.shape == want.shape, (part, key)
                assert got.tobytes() == want.tobytes(), (part, key)
            else:
                assert got == want, (part, key)
