"""bench.py on the host: the reference arm (the fp64 oracle timed on the CPU cores)
prints one JSON line with the keys the benchmark contract asks for, for the forward
workload and for the training workload.  No GPU is needed."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("workload,metric_start", [("large_g_bf16", "slice+deslice"), ("train_bf16", "train step")])
def test_reference_arm_prints_the_contract_line(workload, metric_start):
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", workload,
                        "--steps", "1", "--warmup", "3", "--ref-points", "128"],
                       capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    line = json.loads(r.stdout.strip().splitlines()[-1])
    for key in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in line, key
    assert line["impl"] == "reference" and line["metric"].startswith(metric_start)
    assert line["value"] > 0 and line["cpu_baseline"]["value"] == line["value"]
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0


def test_named_workload_dtype_override():
    """make_named's dtype_override keeps the recipe and changes only the inputs' dtype:
    fp32 inputs are the same draws without the bf16 rounding."""
    sys.path.insert(0, ROOT)
    from paper_2609_32525_gb300.workloads import bf16_round, make_named

    a = make_named("train_bf16", n_override=256)
    b = make_named("train_bf16", n_override=256, dtype_override="f32")
    assert a.dtype == "bf16" and b.dtype == "f32"
    assert (a.B, a.N, a.H, a.d, a.G) == (b.B, b.N, b.H, b.d, b.G)
    for ta, tb in ((a.x_mid, b.x_mid), (a.fx, b.fx), (a.dout, b.dout)):
        assert not (tb == bf16_round(tb)).all()  # fp32 draws carry bits bf16 drops
        assert (ta == bf16_round(tb)).all()      # and round to the bf16 workload's inputs
    assert (a.W_slice == b.W_slice).all() and (a.M == b.M).all()
    with pytest.raises(ValueError):
        make_named("train_bf16", n_override=256, dtype_override="f16")
