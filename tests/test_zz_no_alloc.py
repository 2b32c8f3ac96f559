"""ordermoe_dispatch_noalloc against ordermoe_dispatch.

The no-allocation variant exists for callers that cannot give the library
device memory (a plugin whose host framework owns all device allocations, a
serving loop that may not call cudaMalloc once running). It must produce
exactly what the workspace variant produces. Two calls in a row, with
different inputs, show that the scratch array it keeps between calls needs no
clearing. This file is collected last so that a run stopping at the first
failure has run every other test first; it also passes alone in a fresh
process.
"""
import numpy as np
import pytest
import torch

from paper_2607_17154_gb300 import binding as B
from paper_2607_17154_gb300 import synth

pytestmark = pytest.mark.gpu

DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)
    B.lib()


def _both(chosen, X, T, k, E, d):
    outs = []
    for variant in ("workspace", "noalloc"):
        off = torch.full((E + 1,), -1, dtype=torch.int32, device=DEV)
        rt = torch.full((T * k,), -1, dtype=torch.int32, device=DEV)
        rof = torch.full((T, k), -1, dtype=torch.int32, device=DEV)
        xp = torch.zeros(T * k, d, dtype=torch.bfloat16, device=DEV)
        if variant == "workspace":
            ws = torch.empty(B.ordermoe_dispatch_workspace_bytes(T, k, E), dtype=torch.uint8,
                             device=DEV)
            B.ordermoe_dispatch(chosen, X, T, k, E, d, off, rt, rof, xp, ws)
        else:
            B.ordermoe_dispatch_noalloc(chosen, X, T, k, E, d, off, rt, rof, xp)
        torch.cuda.synchronize()
        outs.append((off.cpu(), rt.cpu(), rof.cpu(), xp.cpu()))
    return outs


def test_noalloc_dispatch_matches_workspace_dispatch_twice_in_a_row():
    rng = np.random.default_rng(77)
    # first call: the largest size allowed (T*k = 262144 entries over 64
    # experts fill the whole fixed scratch array); then a full-size Mixtral
    # batch, then fewer chunks and experts, so stale histogram entries of the
    # earlier calls remain in the shared scratch array
    for T, k, E, d in [(32768, 8, 64, 64), (4096, 2, 8, 4096), (1000, 6, 64, 256), (37, 3, 5, 64)]:
        chosen = torch.as_tensor(rng.integers(0, E, (T, k)).astype(np.int32)).to(DEV)
        X = synth.normal((T, d), 1.0, seed=T + d, device=DEV)
        (a, b) = _both(chosen, X, T, k, E, d)
        for name, u, v in zip(("offsets", "row_token", "row_of", "X_perm"), a, b):
            assert torch.equal(u, v), name
    code, detail = B.ordermoe_device_error()
    assert code == 0, (code, detail)


def test_noalloc_dispatch_rejects_sizes_beyond_its_fixed_scratch():
    T, k, E, d = 131073, 2, 8, 8           # 262146 entries > 262144
    z = torch.empty(0, dtype=torch.int32, device=DEV)
    with pytest.raises(B.OrderMoEError) as ei:
        B.ordermoe_dispatch_noalloc(z, torch.empty(0, dtype=torch.bfloat16, device=DEV), T, k, E, d,
                                    torch.empty(E + 1, dtype=torch.int32, device=DEV), z, z,
                                    torch.empty(0, dtype=torch.bfloat16, device=DEV))
    assert ei.value.code == B.ERR_UNSUPPORTED_SHAPE
    assert "262144" in str(ei.value)
