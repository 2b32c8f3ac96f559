"""CPU-side checks of the C ABI: the library builds for sm_103a, loads
without a GPU, and exports every entry point that include/*.h declares."""
import ctypes
import glob
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_symbols():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names |= set(re.findall(r"\b(ordermoe_\w+)\s*\(", text))
    return sorted(names)


@pytest.fixture(scope="module")
def libpath():
    from paper_2607_17154_gb300 import build
    return build.build()


def test_header_declares_the_hot_path_calls():
    names = declared_symbols()
    for n in ("ordermoe_route_select", "ordermoe_dispatch", "ordermoe_expert_ffn",
              "ordermoe_combine", "ordermoe_build_tables"):
        assert n in names


def test_library_exports_every_declared_symbol(libpath):
    lib = ctypes.CDLL(libpath)
    missing = [n for n in declared_symbols() if not hasattr(lib, n)]
    assert not missing, missing
    out = subprocess.run(["nm", "-D", "--defined-only", libpath], capture_output=True, text=True).stdout
    exported = set(l.split()[-1] for l in out.splitlines() if l.strip())
    assert set(declared_symbols()) <= exported


def test_header_compiles_as_plain_c(tmp_path):
    src = tmp_path / "t.c"
    src.write_text('#include "ordermoe.h"\nint main(void){return ORDERMOE_OK;}\n')
    r = subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-I", os.path.join(ROOT, "include"),
                        "-c", str(src), "-o", str(tmp_path / "t.o")], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_size_queries_without_gpu(libpath):
    from paper_2607_17154_gb300 import binding as B
    assert B.ordermoe_version() >= 100
    assert B.ordermoe_tables_bytes(8, 4) >= 832 + 2 * 4 * 64 + 4 * 64
    assert B.ordermoe_tables_bytes(65, 4) == 0 and B.ordermoe_tables_bytes(8, 33) == 0
    assert B.ordermoe_dispatch_workspace_bytes(4096, 2, 8) >= 32 * 8 * 4
    assert B.ordermoe_dispatch_workspace_bytes(10, 2, 65) == 0


def test_no_cluster_multicast_copies_in_the_kernels():
    """No bulk copy in the library carries .multicast::cluster: bench.py's
    replicas run the same kernels on every GPU of a node, so every CTA loads
    its own boxes. (The tcgen05.commit arrive on both CTAs of a pair is a
    barrier signal, not a copy, and may multicast.)"""
    csrc = os.path.join(ROOT, "paper_2607_17154_gb300", "csrc")
    bad, copies = [], 0
    for path in sorted(glob.glob(os.path.join(csrc, "*.cu")) + glob.glob(os.path.join(csrc, "*.cuh"))):
        text = open(path).read()
        # PTX strings are split over adjacent literals: join each asm statement first
        for stmt in re.findall(r"asm\s+volatile\s*\((.*?)\);", text, flags=re.S):
            ptx = "".join(re.findall(r'"((?:[^"\\]|\\.)*)"', stmt))
            copies += "cp.async.bulk" in ptx
            if "cp.async.bulk" in ptx and "multicast::cluster" in ptx:
                bad.append((os.path.basename(path), ptx[:80]))
    assert copies > 0 and not bad, (copies, bad)
