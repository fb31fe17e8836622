"""bench.py's byte accounting for each kind of step (CPU only): the algorithmic bytes per
parameter behind the roofline figures."""
import pytest

import bench


@pytest.mark.parametrize("K", [1, 2, 4, 8, 16])
def test_bytes_per_parameter(K):
    # pass 1: K replicas read, the mean written over replica 0 (K > 1); LARS also reads w
    assert bench.pass1_bytes_per_param(K) == 4 * K + (4 if K > 1 else 0)
    assert bench.pass1_bytes_per_param(K, read_w=True) == bench.pass1_bytes_per_param(K) + 4
    # pass 2: gbar, w, m read; w, m written
    assert bench.pass2_bytes_per_param() == 20
    assert bench.pass2_bytes_per_param(with_momentum=False) == 12
    # the step as built, and the least any design must move
    assert bench.step_design_bytes_per_param(K) == bench.pass1_bytes_per_param(K) + 20
    assert bench.step_min_bytes_per_param(K) == 4 * K + 16
    assert bench.step_min_bytes_per_param(K, read_w=True) == 4 * K + 20
    assert bench.step_min_bytes_per_param(K) <= bench.step_design_bytes_per_param(K)
    # no momentum buffer: m is neither read nor written; a per-element gradscale is read
    assert bench.pass2_bytes_per_param(False, True) == 16
    assert bench.step_min_bytes_per_param(K, with_momentum=False) == 4 * K + 8
    assert bench.step_min_bytes_per_param(K, per_element=True) == 4 * K + 20
    assert bench.step_design_bytes_per_param(K, False, False, True) == \
        bench.pass1_bytes_per_param(K) + 16
    assert bench.scale_elem_bytes_per_param() == 12


def test_step_kinds():
    # only LARS reads w in pass 1; only the refresh kind refreshes the gradscale every step
    assert bench.STEP_KINDS == {"ags": (False, False), "refresh": (False, True),
                                "lars": (True, False), "update-scale": (False, False),
                                "sharded": (False, False)}
    assert set(bench.STEP_KIND_TEXT) == set(bench.STEP_KINDS)


@pytest.mark.parametrize("kind", ["ags", "lars"])
def test_reference_arm_prints_the_contract_line(kind):
    """`bench.py --impl reference` (the oracle on the host) prints one JSON line with the keys
    the benchmark contract asks for, on the same metric and unit as the GPU arm."""
    import json
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    out = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference",
                          "--workload", "resnet20", "--steps", "1", "--warmup", "0",
                          "--step-kind", kind],
                         capture_output=True, text=True, timeout=300, cwd=root)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [ln for ln in out.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["unit"] == bench.UNIT
    assert d["value"] > 0 and d["higher_is_better"] is True and d["n_gpus"] == 1
    assert d["steps"] == 1 and d["warmup"] == 0 and d["vs_baseline"] is None
    assert d["config"]["workload"].startswith("resnet20")
    assert d["config"]["step"] == bench.STEP_KIND_TEXT[kind]
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert cb["cores"] == min(os.cpu_count(), bench.host_cores()) and cb["host_cpu_count"] == os.cpu_count()
    assert d["e2e"] == {"value": d["value"], "unit": bench.UNIT, "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}
