"""The C-ABI library builds, loads without a GPU, and exports every entry point
that include/*.h declares.  No compute call is made here."""
import ctypes
import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = []
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        names += re.findall(r"\b(maps_[a-z0-9_]+)\s*\(", text)
    return sorted(set(names))


@pytest.fixture(scope="module")
def libmaps():
    from paper_2609_15359_gb300 import build
    path = build.build()
    return ctypes.CDLL(path)


def test_header_declares_the_four_calls():
    names = declared_functions()
    for n in ("maps_calibrate", "maps_project_occupancy", "maps_dispatch", "maps_order_local"):
        assert n in names


def test_library_exports_every_declared_symbol(libmaps):
    missing = [n for n in declared_functions() if not hasattr(libmaps, n)]
    assert not missing, missing


def test_binding_loads_and_host_only_queries(libmaps):
    from paper_2609_15359_gb300 import maps as M
    assert set(M.EXPORTS) <= set(declared_functions())
    assert M.lib.maps_version() == 100
    # workspace queries are host arithmetic only
    assert M.lib.maps_calibrate_workspace_size(10**6, 10**6) > 0
    assert M.lib.maps_project_occupancy_workspace_size(256, 65536, 2**20) >= 256
    big = M.lib.maps_dispatch_workspace_size(M.MODE_SNAPSHOT, 256, 65536, 65536)
    assert big > 2 * 256 * 1024 * 4  # look-back state for every tile and decoder
    assert M.lib.maps_order_local_workspace_size(10**6, 256) > 10**6 * 24


def test_static_order_array_holds_its_largest_calls(libmaps):
    """maps_order_local_static takes up to 65,536 entries and 4,096 decoders in
    a fixed 5 MiB array: the workspace those calls need fits it, and a queue of
    all 65,536 entries has room for its sixteen runs' pairwise ranks."""
    from paper_2609_15359_gb300 import maps as M
    for D in (1, 7, 256, 1024, 1025, 4096):
        assert M.lib.maps_order_local_workspace_size(65536, D) <= 5 << 20
    small = M.lib.maps_order_local_workspace_size(65536, 1)
    assert small > 15 * 14 * 4608 * 2  # 210 run pairs of 16-bit counts
