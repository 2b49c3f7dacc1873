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


# Values for the placeholders the documentation writes in place of a number or a name.
_PLACEHOLDER = {"--gpus": "2", "--steps": "1", "--warmup": "3", "--variant": "frozen"}


def _documented_bench_commands():
    """The bench.py argument lists in the fenced code blocks of the README and the
    profile summaries (up to the first shell operator, comment or closing quote)."""
    import glob
    import re
    import shlex

    files = [os.path.join(ROOT, "README.md")] + sorted(glob.glob(os.path.join(ROOT, "profiles", "*.md")))
    cmds = []
    for path in files:
        fenced = False
        for line in open(path, encoding="utf-8"):
            if line.lstrip().startswith("```"):
                fenced = not fenced
                continue
            if not fenced:
                continue
            for m in re.finditer(r"bench\.py((?:\s+[^\s\"'`>|&#;)]+)*)", line):
                argv = shlex.split(m.group(1))
                cmds.append((os.path.relpath(path, ROOT), [
                    _PLACEHOLDER.get(argv[i - 1], a) if i and re.fullmatch(r"[A-Z]", a) else a
                    for i, a in enumerate(argv)]))
    return cmds


def test_documented_bench_commands_parse():
    """Every bench.py command that the README and profiles/ give parses with the
    current flags, so the recipes beside the committed numbers still run."""
    import bench
    from paper_2609_32525_gb300.workloads import NAMED

    cmds = _documented_bench_commands()
    assert len(cmds) >= 8
    parser = bench.build_parser()
    for path, argv in cmds:
        try:
            args = parser.parse_args(argv)
        except SystemExit:
            pytest.fail(f"{path}: bench.py {' '.join(argv)} does not parse")
        assert args.workload in NAMED, f"{path}: unknown workload {args.workload}"
