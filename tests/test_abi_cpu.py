"""The C ABI on the host (no GPU): exports, defaults, workspace sizing, the chunk
plan, and argument validation (which returns before any CUDA call)."""
import ctypes
import json
import math
import os

import pytest

from paper_2603_18112_gb300 import build as B
from paper_2603_18112_gb300 import tula_ags as T
from paper_2603_18112_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_hparams.json")


@pytest.fixture(scope="module")
def lib():
    B.build()
    return T.lib()


def test_every_declared_function_is_exported(lib):
    names = T.header_functions()
    assert "tula_ags_step" in names and "tula_layer_stats" in names
    for name in names:
        assert hasattr(lib, name), name


def test_defaults_match_paper(lib):
    gold = json.load(open(GOLDEN))
    for K in (1, 4, 8, 16):
        hp = T.tula_ags_default_hparams(K)
        assert hp.K == K
        assert hp.rule == T.TULA_RULE_AGS and hp.granularity == T.TULA_SCALE_PER_TENSOR
        assert hp.delta == gold["delta"]["value"]
        assert hp.eps == pytest.approx(gold["eps"]["value"], rel=1e-7)
        assert hp.s_max == pytest.approx(math.sqrt(K), rel=1e-7)  # sqrt(b_large / b_small)
        assert not hp.scale and not hp.state and not hp.workspace


@pytest.mark.parametrize("pass_,stage_kb,streams", [(1, 36, s) for s in (1, 2, 3, 4, 9, 17, 18)]
                         + [(2, 24, s) for s in (2, 3, 4)]
                         + [(3, 45, s) for s in (2, 3, 5, 9, 17)])
def test_tile_fits_one_stage(lib, pass_, stage_kb, streams):
    C = T.tula_ags_chunk_elems(pass_, streams)
    stage = stage_kb * 1024
    assert C % 128 == 0 and 0 < C * 4 * streams <= stage
    assert C * 4 * streams > stage - 128 * 4 * streams  # the largest multiple of 128 that fits


def test_tile_sizes_reject_bad_arguments(lib):
    for pass_, streams in ((1, 0), (1, 19), (2, 0), (2, 5), (0, 2), (3, 0), (3, 19), (4, 2)):
        assert T.lib().tula_ags_chunk_elems(pass_, streams) == T.TULA_ERR_ARG


@pytest.mark.parametrize("streams", [1, 9])
def test_plan_covers_every_element_once(lib, streams):
    C = T.tula_ags_chunk_elems(1, streams)
    numels = [0, 1, 3, C - 1, C, C + 1, 5 * C + 7, 64]
    starts = T.tula_ags_plan_chunks(numels, C)
    assert starts[0] == 0
    for p, n in enumerate(numels):
        nch = starts[p + 1] - starts[p]
        assert nch == max(1, math.ceil(n / C))
        covered = sum(min(C, n - i * C) for i in range(nch)) if n else 0
        assert covered == n
    assert starts == T.tula_ags_plan_chunks(numels, C)  # depends on the numels only


def test_workspace_size_depends_on_the_tensor_count_only(lib):
    """Norms accumulate per tensor (exact integer accumulators), not per tile: the workspace
    grows with the number of tensors and does not change with their sizes or with K."""
    ps = W.param_set("resnet50")
    a = T.tula_ags_workspace_size(ps.numels, 8)
    assert a > 0 and a % 256 == 0
    assert T.tula_ags_workspace_size([n * 1000 for n in ps.numels], 8) == a
    assert T.tula_ags_workspace_size(ps.numels, 1) == a == T.tula_ags_workspace_size(ps.numels, 16)
    assert T.tula_ags_workspace_size(ps.numels + [10], 8) > a


@pytest.mark.parametrize("numels,K", [([], 1), ([3, -1], 1), ([3], 0), ([3], 17)])
def test_workspace_size_rejects(lib, numels, K):
    with pytest.raises(T.TulaError) as e:
        T.tula_ags_workspace_size(numels, K)
    assert e.value.code == T.TULA_ERR_ARG


@pytest.mark.parametrize("K", [1, 2, 4, 8, 16])
def test_size_limit(lib, K):
    """All tensors together may span fewer than 2^31 tiles of either pass at its smallest tile
    (the header's stated limit); the check happens before any launch."""
    tile = min(T.tula_ags_chunk_elems(1, K + 2 if K == 1 else K + 1), T.tula_ags_chunk_elems(2, 4))
    limit = (2 ** 31 - 1) * tile
    half = 2 ** 30 * tile  # split at a tile boundary: 2^30 + (2^30 - 1) tiles
    assert T.tula_ags_workspace_size([limit], K) > 0
    assert T.tula_ags_workspace_size([half, limit - half], K) > 0
    for numels in ([limit + 1], [half, limit - half + 1]):
        with pytest.raises(T.TulaError) as e:
            T.tula_ags_workspace_size(numels, K)
        assert e.value.code == T.TULA_ERR_ARG


def _call_step(lib, n=2, K=1, params=None, grads=None, moms=None, numels=None, hp=None,
               momentum=0.9):
    P = ctypes.c_void_p
    fake = [0x10000 * (i + 1) for i in range(64)]  # aligned, never dereferenced on error paths
    params = params if params is not None else fake[:n]
    grads = grads if grads is not None else fake[8:8 + K * n]
    numels = numels if numels is not None else [5] * n
    pa = (P * max(1, len(params)))(*params)
    ga = (P * max(1, len(grads)))(*grads)
    ma = None if moms == "null" else (P * n)(*(moms or fake[40:40 + n]))
    na = (ctypes.c_int64 * max(1, len(numels)))(*numels)
    if hp is None:
        hp = T.tula_ags_default_hparams(K)
        hp.scale = 0x20000
        hp.state = 0x30000
        hp.workspace = 0x40000
        hp.workspace_bytes = 1 << 30
    return lib.tula_ags_step(pa, ga, ma, na, len(numels), 0.1, momentum, 0.0,
                             ctypes.byref(hp), None)


def test_step_argument_errors(lib):
    assert _call_step(lib, numels=[]) == T.TULA_ERR_ARG                 # n_tensors < 1
    assert _call_step(lib, numels=[5, -2]) == T.TULA_ERR_ARG           # negative numel
    assert _call_step(lib, params=[0x10000, 0]) == T.TULA_ERR_ARG      # NULL param
    assert _call_step(lib, params=[0x10000, 0x10002]) == T.TULA_ERR_ARG  # not 4-byte aligned
    assert _call_step(lib, moms="null") == T.TULA_ERR_ARG              # momentum without buffer
    hp = T.tula_ags_default_hparams(1)
    assert _call_step(lib, hp=hp) == T.TULA_ERR_ARG                    # no state / scale
    for field, bad in (("K", 0), ("K", 17), ("rule", 9), ("granularity", 5), ("force_branch", 7)):
        hp = T.tula_ags_default_hparams(1)
        hp.scale, hp.state, hp.workspace, hp.workspace_bytes = 0x20000, 0x30000, 0x40000, 1 << 30
        setattr(hp, field, bad)
        assert _call_step(lib, hp=hp) == T.TULA_ERR_ARG, field
    hp = T.tula_ags_default_hparams(1)
    hp.scale, hp.state, hp.workspace, hp.workspace_bytes = 0x20000, 0x30000, 0x40000, 1 << 30
    hp.refresh_scale = 1                                                # K = 1 has no g_small
    assert _call_step(lib, hp=hp) == T.TULA_ERR_ARG
    hp = T.tula_ags_default_hparams(2)
    hp.scale, hp.state, hp.workspace, hp.workspace_bytes = 0x20000, 0x30000, 0x40000, 16
    assert _call_step(lib, K=2, hp=hp) == T.TULA_ERR_WORKSPACE          # too small
    hp.workspace_bytes, hp.workspace = 1 << 30, 0x40010
    assert _call_step(lib, K=2, hp=hp) == T.TULA_ERR_WORKSPACE          # not 256-byte aligned
    hp.workspace = 0
    assert _call_step(lib, K=2, hp=hp) == T.TULA_ERR_WORKSPACE


def test_error_strings(lib):
    for code in (0, -1, -2, -3, -4, 99):
        assert isinstance(T.tula_ags_error_string(code), str)
    assert T.tula_ags_last_cuda_error() == 0


def test_binding_refuses_replica_lists_that_do_not_match(lib):
    """The wrappers check the list lengths before the C call: the library reads hp.K * n
    gradient pointers and n momentum pointers, so a shorter list must never reach it."""
    import torch
    params = [torch.zeros(4), torch.zeros(4)]
    grads = [[torch.zeros(4), torch.zeros(4)]]
    hp = T.tula_ags_default_hparams(2)                       # K = 2, one replica list given
    for fn in (T.tula_ags_step, T.tula_ags_step_static_scratch):
        with pytest.raises(ValueError, match="replica"):
            fn(params, grads, params, 0.1, 0.9, 0.0, hp)
        hp1 = T.tula_ags_default_hparams(1)
        with pytest.raises(ValueError, match="tensors"):     # replica 0 short of one tensor
            fn(params, [[torch.zeros(4)]], params, 0.1, 0.9, 0.0, hp1)
        with pytest.raises(ValueError, match="momentum"):
            fn(params, grads, params[:1], 0.1, 0.9, 0.0, hp1)
    with pytest.raises(ValueError):
        T.AGSOptimizerStep(params, [[torch.zeros(4)]])
    with pytest.raises(ValueError):
        T.AGSOptimizerStep(params, [])


def test_sharded_step_argument_errors(lib):
    """The two halves of a sharded step check their arguments like tula_ags_step, and the share
    pointer (NULL or not 8-byte aligned) before any CUDA call."""
    P = ctypes.c_void_p
    ptrs = (P * 4)(*[0x10000 * (i + 1) for i in range(4)])
    numels = (ctypes.c_int64 * 2)(5, 7)
    hp = T.tula_ags_default_hparams(1)
    hp.scale, hp.state, hp.workspace, hp.workspace_bytes = 0x20000, 0x30000, 0x40000, 1 << 30
    for share in (None, 0x50004):
        assert lib.tula_ags_shard_reduce(ptrs, ptrs, ptrs, numels, 2, 0.9, ctypes.byref(hp),
                                         share, None) == T.TULA_ERR_ARG
        assert lib.tula_ags_shard_update(ptrs, ptrs, ptrs, numels, 2, 0.1, 0.9, 0.0,
                                         ctypes.byref(hp), share, None) == T.TULA_ERR_ARG
    hp.state = 0
    assert lib.tula_ags_shard_reduce(ptrs, ptrs, ptrs, numels, 2, 0.9, ctypes.byref(hp),
                                     0x50000, None) == T.TULA_ERR_ARG


def test_plan_argument_errors_come_before_any_cuda_call(lib):
    """tula_ags_plan_create checks the sizes and every pointer before it asks CUDA for the
    current device, and tula_ags_plan_step refuses a NULL plan or hp; no GPU is needed to see
    TULA_ERR_ARG, and *plan_out stays NULL on every error."""
    P = ctypes.c_void_p
    ptrs = (P * 4)(*[0x100000 * (i + 1) for i in range(4)])
    numels = (ctypes.c_int64 * 2)(5, 7)
    hp = T.tula_ags_default_hparams(2)
    out = P(0x1234)
    create = lib.tula_ags_plan_create
    assert create(ptrs, ptrs, ptrs, numels, 2, ctypes.byref(hp), None) == T.TULA_ERR_ARG
    assert create(ptrs, ptrs, ptrs, numels, 2, None, ctypes.byref(out)) == T.TULA_ERR_ARG
    assert out.value is None
    bad = (P * 4)(0x100000, 0x100002, 0x100000, 0x100000)     # misaligned second gradient
    assert create(ptrs, bad, ptrs, numels, 2, ctypes.byref(hp), ctypes.byref(out)) == T.TULA_ERR_ARG
    nul = (P * 4)(0x100000, None, 0x100000, 0x100000)          # a missing momentum buffer
    assert create(ptrs, ptrs, nul, numels, 2, ctypes.byref(hp), ctypes.byref(out)) == T.TULA_ERR_ARG
    hp.K = 0
    assert create(ptrs, ptrs, ptrs, numels, 2, ctypes.byref(hp), ctypes.byref(out)) == T.TULA_ERR_ARG
    hp.K = 2
    neg = (ctypes.c_int64 * 2)(5, -1)
    assert create(ptrs, ptrs, ptrs, neg, 2, ctypes.byref(hp), ctypes.byref(out)) == T.TULA_ERR_ARG
    assert out.value is None
    assert lib.tula_ags_plan_step(None, 0.1, 0.9, 0.0, ctypes.byref(hp), None) == T.TULA_ERR_ARG
    assert lib.tula_ags_plan_destroy(None) == T.TULA_OK
    assert "allocation" in T.tula_ags_error_string(T.TULA_ERR_NO_MEMORY)


def test_plan_binding_checks_replica_lists(lib):
    """The wrapper refuses replica and momentum lists that do not match hp.K and the tensor
    count, before the C call (which reads K * n gradient pointers)."""
    import torch
    params = [torch.zeros(4), torch.zeros(4)]
    hp = T.tula_ags_default_hparams(2)
    with pytest.raises(ValueError, match="replica"):
        T.tula_ags_plan_create(params, [params], params, hp)
    with pytest.raises(ValueError, match="momentum"):
        T.tula_ags_plan_create(params, [params, params], params[:1], hp)
