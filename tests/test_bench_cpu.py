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


def test_step_kinds():
    # only LARS reads w in pass 1; only the refresh kind refreshes the gradscale every step
    assert bench.STEP_KINDS == {"ags": (False, False), "refresh": (False, True),
                                "lars": (True, False)}
    assert set(bench.STEP_KIND_TEXT) == set(bench.STEP_KINDS)
