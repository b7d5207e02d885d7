"""Host-side logic of bench.py that needs no GPU: the staging arena of the
end-to-end path and the traffic table's source keys."""
import os

import numpy as np
import pytest

import bench
from paper_2609_15359_gb300 import workloads as W


@pytest.mark.parametrize("name", ["tiny", "d16", "large"])
def test_input_arena_layout(name):
    w = W.make(name)
    fields, total, copy_bytes = bench.input_layout(w)
    R, J = w["R"], w["J"]
    spans = []
    for k, (off, count, dt) in fields.items():
        assert off % 256 == 0, k  # every field starts 256-byte aligned
        spans.append((off, off + count * np.dtype(dt).itemsize, k))
    spans.sort()
    for (a0, a1, ka), (b0, b1, kb) in zip(spans, spans[1:]):
        assert a1 <= b0, (ka, kb)  # no two fields overlap
    assert spans[-1][2] == "dec_all" and spans[-1][1] <= total
    # one copy covers every input and the residents' decoders, not the choices
    dec_off = fields["dec_all"][0]
    assert copy_bytes == dec_off + 4 * R
    assert all(off + count * np.dtype(dt).itemsize <= copy_bytes
               for k, (off, count, dt) in fields.items() if k != "dec_all")
    arrays = bench.input_arrays(w)
    assert set(arrays) == set(fields)
    for k, a in arrays.items():
        assert len(a) == fields[k][1], k
    assert np.array_equal(arrays["dec_all"][:R], w["res_dec"])
    assert not arrays["dec_all"][R:].any() and len(arrays["dec_all"]) == R + J


def test_traffic_table_keys_existing_sources():
    for call, t in bench.TRAFFIC.items():
        src = os.path.join(bench.ROOT, "paper_2609_15359_gb300", "csrc", t["source"])
        assert os.path.exists(src), call
        assert call in bench.KERNELS
        # a figure is only reported for the source it was measured on
        assert bench.traffic_for(call) in (None, t["bytes"])
