"""Host-side logic of bench.py that needs no GPU: the staging arena of the
end-to-end path, the traffic table's source keys and the reference arm (the
oracle, timed on the host)."""
import argparse
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


def test_oracle_step_runs_the_whole_workload_and_matches_tier_b():
    """The CPU baseline's step runs every part of the path on the whole
    workload; on the tiny workload its dispatch equals the by-definition
    oracle's."""
    import oracle as O
    w = W.make("tiny")
    step = bench.OracleStep(w)
    assert step.run() > 0.0
    q = O.calibrate(w["cal_true"], w["cal_pred"], w["alphas_ppm"][0])[1]
    U = O.bound(np.concatenate([w["res_pred"], w["cand_pred"]]), q)[1]
    R = w["R"]
    _, K = O.occupancy(w["D"], w["H"], w["res_off"], w["res_prompt"], w["res_gen"], U[:R])
    assert np.array_equal(step.K, K)
    secs, used = bench.time_oracle(step, 2, 2, warm=0)
    assert secs > 0.0 and used >= 1
    O.p_threads(1)


def test_reference_arm_json_line(monkeypatch):
    monkeypatch.setattr(bench, "WORKLOAD", "d16")
    args = argparse.Namespace(steps=2, warmup=1, gpus=1, impl="reference")
    assert bench.bench_reference(args, 2, 1) is None  # other ranks do no work
    r = bench.bench_reference(args, 1, 0)
    assert r["impl"] == "reference" and r["value"] > 0 and r["unit"] == bench.UNIT
    assert r["steps"] == 2 and r["warmup"] == 1 and r["higher_is_better"] is True
    assert r["ms_per_step"] > 0 and r["metric"] == bench.METRIC
    cb = r["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == r["value"]
    assert cb["sample"] and "whole steps" in cb["sample"]
    assert r["e2e"] == {"value": r["value"], "unit": r["unit"], "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}


def test_calibration_report_reaches_the_coverage_target(oracle):
    """The bench's underestimation report on Large's held-out candidates, with
    the oracle's quantile: the calibrated bound underestimates at most about
    alpha of them (three standard errors of slack), the raw prediction far
    more."""
    import bench
    from paper_2609_15359_gb300 import workloads as W
    w = W.make("large")
    st, q = oracle.calibrate(w["cal_true"], w["cal_pred"], w["alphas_ppm"][0])
    assert st == 0
    r = bench.calibration_report(w, int(q))
    a, n = r["alpha"], r["held_out"]
    assert r["under_calibrated"] <= a + 3 * (a * (1 - a) / n) ** 0.5
    assert r["under_raw"] > 2 * a and r["under_pred_x1.1"] > r["under_calibrated"]
