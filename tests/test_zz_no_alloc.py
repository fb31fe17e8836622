"""The allocation-free step, tula_ags_step_static_scratch.

It serves callers that may not allocate device memory: code inside a host
framework that owns every device allocation, latency-critical loops where
cudaMalloc's implicit device synchronization is not acceptable, and plain C
callers with no place to keep a workspace between calls.  Its scratch is a
static device array inside the library, so it must give exactly what
tula_ags_step gives with a caller-provided workspace -- also on the second call
in a row, when the array still holds the first call's contents.

This file is collected last, so a run that stops at its first failure has run
every other test before it.
"""
import ctypes

import numpy as np
import pytest
import torch

from _parity import assert_f32_close, assert_norm_close, assert_state_close
from paper_2603_18112_gb300 import build as B
from paper_2603_18112_gb300 import tula_ags as T
from paper_2603_18112_gb300 import workloads as W


def test_rejects_tensor_lists_beyond_the_static_scratch():
    """Host-only: a list needing more than TULA_STATIC_SCRATCH_BYTES is refused before any
    CUDA call (the pointers below are never dereferenced)."""
    B.build()
    lib = T.lib()
    n = 11000  # about 1.6 KB of scratch per tensor: 17.3 MB, beyond 16 MiB
    numels = [5] * n
    assert T.tula_ags_workspace_size(numels, 1) > T.TULA_STATIC_SCRATCH_BYTES
    assert T.tula_ags_workspace_size(numels[:10600], 1) <= T.TULA_STATIC_SCRATCH_BYTES
    P = ctypes.c_void_p
    ptrs = (P * n)(*[0x100000 * (i + 1) for i in range(n)])
    hp = T.tula_ags_default_hparams(1)
    hp.scale, hp.state = 0x200000, 0x300000
    rc = lib.tula_ags_step_static_scratch(ptrs, ptrs, ptrs, (ctypes.c_int64 * n)(*numels), n,
                                          0.1, 0.9, 0.0, ctypes.byref(hp), None)
    assert rc == T.TULA_ERR_SCRATCH_LIMIT
    assert "static scratch" in T.tula_ags_error_string(rc)


def test_argument_errors_come_before_any_cuda_call():
    """Host-only: every argument check of tula_ags_step runs before the static-scratch call
    looks up its array or enqueues its memsets.  Without a GPU any CUDA call would fail with
    TULA_ERR_CUDA, so TULA_ERR_ARG here shows that nothing reached CUDA."""
    B.build()
    lib = T.lib()
    P = ctypes.c_void_p
    ptrs = (P * 4)(*[0x100000 * (i + 1) for i in range(4)])
    numels = (ctypes.c_int64 * 2)(5, 7)
    hp = T.tula_ags_default_hparams(1)
    hp.scale = 0x200000                                    # hp.state left NULL
    rc = lib.tula_ags_step_static_scratch(ptrs, ptrs, ptrs, numels, 2, 0.1, 0.9, 0.0,
                                          ctypes.byref(hp), None)
    assert rc == T.TULA_ERR_ARG
    hp.state, hp.rule = 0x300000, 9                        # bad enum
    assert lib.tula_ags_step_static_scratch(ptrs, ptrs, ptrs, numels, 2, 0.1, 0.9, 0.0,
                                            ctypes.byref(hp), None) == T.TULA_ERR_ARG
    hp.rule = T.TULA_RULE_AGS
    bad = (P * 4)(0x100000, 0x100002, 0x100000, 0x100000)  # misaligned second tensor
    assert lib.tula_ags_step_static_scratch(bad, ptrs, ptrs, numels, 2, 0.1, 0.9, 0.0,
                                            ctypes.byref(hp), None) == T.TULA_ERR_ARG
    assert lib.tula_ags_static_scratch_error(None, None) == T.TULA_ERR_ARG


def _model(wl, K, pset):
    buf = W.allocate(wl, "cuda", K=K, pset=pset)
    W.fill_state(buf, wl)
    return buf


@pytest.mark.gpu
def test_static_scratch_step_matches_workspace_step():
    B.build()
    T.lib()
    ps = W.param_set("resnet20")
    for n in (0, 1, 5, 16383, 16385, 100003):   # empty, tiny and ragged-chunk tensors too
        ps.add((n,), W.KIND_NORMAL)
    wl = W.workload("resnet50", seed=77)
    K = 4
    ref = _model(wl, K, ps)
    new = _model(wl, K, ps)
    n = ps.n_tensors

    ref_step = T.AGSOptimizerStep(ref.w, ref.g, ref.m, s_max=2.0)      # caller workspace

    hp = T.tula_ags_default_hparams(K)                                  # no workspace at all
    scale = torch.ones(n, dtype=torch.float32, device="cuda")
    state = torch.zeros(T.TULA_STATE_LEN, dtype=torch.float64, device="cuda")
    stats = torch.zeros(n, T.TULA_STATS_LEN, dtype=torch.float64, device="cuda")
    hp.s_max = 2.0
    hp.scale, hp.state, hp.layer_stats = scale.data_ptr(), state.data_ptr(), stats.data_ptr()

    for call, refresh in ((1, True), (2, False)):  # two calls in a row; the 2nd is scaled
        for buf in (ref, new):
            W.fill_grads(buf, wl, step=1)
        ref_step.step(wl.lr, wl.momentum, wl.weight_decay, refresh_scale=refresh)
        hp.refresh_scale = 1 if refresh else 0
        T.tula_ags_step_static_scratch(new.w, new.g, new.m, wl.lr, wl.momentum,
                                       wl.weight_decay, hp)
        torch.cuda.synchronize()
        where = f"call {call}"
        assert torch.equal(new.g_flats[0], ref.g_flats[0]), where + ": replica mean"
        assert_f32_close(new.w_flat.cpu().numpy(), ref.w_flat.cpu().numpy(), where + " w")
        assert_f32_close(new.m_flat.cpu().numpy(), ref.m_flat.cpu().numpy(), where + " m")
        assert_state_close(state.cpu().numpy(), ref_step.state.cpu().numpy(), where + " state")
        for c in range(T.TULA_STATS_LEN):
            assert_norm_close(stats[:, c].cpu().numpy(), ref_step.stats[:, c].cpu().numpy(),
                              f"{where} stats col {c}")
        assert_norm_close(scale.cpu().numpy(), ref_step.scale.cpu().numpy(), where + " scale")
    assert state[3].item() == 1.0  # TULA_STATE_SCALED: the second call took the scaled branch
    assert np.isfinite(stats.cpu().numpy()).all()


@pytest.mark.gpu
def test_static_scratch_reports_a_wait_that_ran_out():
    """Failure detection on the static scratch, without a fault: the bounded-wait check runs
    out against the static array's error word (about two seconds), the word survives the next
    static-scratch step (its memsets leave it alone), tula_ags_static_scratch_error reads bit 0
    and clears it, and the step after that still matches tula_ags_step."""
    B.build()
    T.lib()
    ps = W.param_set("resnet20")
    ps.add((40000,), W.KIND_NORMAL)
    wl = W.workload("resnet50", seed=78)
    K = 2
    ref = _model(wl, K, ps)
    new = _model(wl, K, ps)
    n = ps.n_tensors
    ref_step = T.AGSOptimizerStep(ref.w, ref.g, ref.m, s_max=2.0)
    hp = T.tula_ags_default_hparams(K)
    scale = torch.ones(n, dtype=torch.float32, device="cuda")
    state = torch.zeros(T.TULA_STATE_LEN, dtype=torch.float64, device="cuda")
    hp.s_max = 2.0
    hp.scale, hp.state = scale.data_ptr(), state.data_ptr()

    def both_steps(seed_step):
        for buf in (ref, new):
            W.fill_grads(buf, wl, step=seed_step)
        ref_step.step(wl.lr, wl.momentum, wl.weight_decay)
        T.tula_ags_step_static_scratch(new.w, new.g, new.m, wl.lr, wl.momentum,
                                       wl.weight_decay, hp)

    torch.cuda.synchronize()
    assert T.tula_ags_static_scratch_error() in (0, 1)  # whatever an earlier test left: cleared
    assert T.tula_ags_static_scratch_error() == 0
    both_steps(1)
    assert T.tula_ags_static_scratch_error() == 0       # every wait of that step completed
    T.tula_ags_static_scratch_check_wait_timeout()
    both_steps(2)                                       # the word stays set through this step
    assert T.tula_ags_static_scratch_error() == 1       # reported ...
    assert T.tula_ags_static_scratch_error() == 0       # ... and cleared by the read
    both_steps(3)
    torch.cuda.synchronize()
    assert T.tula_ags_static_scratch_error() == 0
    assert torch.equal(new.g_flats[0], ref.g_flats[0]), "replica mean"
    assert_f32_close(new.w_flat.cpu().numpy(), ref.w_flat.cpu().numpy(), "w")
    assert_f32_close(new.m_flat.cpu().numpy(), ref.m_flat.cpu().numpy(), "m")
    assert_state_close(state.cpu().numpy(), ref_step.state.cpu().numpy(), "state")
    assert state[1].item() == 3.0
