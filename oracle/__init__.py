"""CPU oracle for the AGS optimizer step -- TEST INFRASTRUCTURE ONLY.

A thin ctypes wrapper over ``tula_oracle.c``: a plain, slow, single-threaded
restatement of the optimizer step of Tula (arXiv 2603.18112) written from the
paper (Eq. 1c, Eq. 5, Eq. 7b, Eq. 8, Algorithm 1, Sec. IV-A/B).  Only the test
suite, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline and
reference legs may import it.  It shares no code with the CUDA library and
never imports it.

Arrays are numpy ``float32`` (tensors) and ``float64`` (state, statistics);
tensors are updated in place, like the library does on the device.

Parity: every function is pinned by ``tests/test_oracle_pins.py`` (closed
forms, brute force, torch.optim.SGD for the unscaled case, hand-worked
examples, invariants); none is "parity unpinned".
"""
from __future__ import annotations

import ctypes
import math
from dataclasses import dataclass

import numpy as np

from ._build import build_oracle

RULE_AGS, RULE_NONE, RULE_LARS, RULE_STATIC = 0, 1, 2, 3
GRAN_TENSOR, GRAN_ELEMENT = 0, 1
BRANCH_AUTO, BRANCH_SCALED, BRANCH_UNSCALED = 0, 1, 2
STATS_LEN = 8
STATE_LEN = 4


class _HP(ctypes.Structure):
    _fields_ = [
        ("K", ctypes.c_int),
        ("rule", ctypes.c_int),
        ("granularity", ctypes.c_int),
        ("force_branch", ctypes.c_int),
        ("refresh_scale", ctypes.c_int),
        ("has_momentum", ctypes.c_int),
        ("delta", ctypes.c_float),
        ("eps", ctypes.c_float),
        ("s_max", ctypes.c_float),
        ("static_s", ctypes.c_float),
        ("lars_trust", ctypes.c_float),
    ]


@dataclass
class OracleHP:
    """AGS hyper-parameters.  Defaults: delta = 0.5 (Sec. III-C, Sec. IV-B),
    eps = 1e-8 (Algorithm 1 input), s_max = sqrt(b_large / b_small) with
    b_small = one replica's share of the large batch, i.e. sqrt(K)
    (Algorithm 1, UpdateGradScale)."""

    K: int = 1
    rule: int = RULE_AGS
    granularity: int = GRAN_TENSOR
    force_branch: int = BRANCH_AUTO
    refresh_scale: bool = False
    has_momentum: bool = True
    delta: float = 0.5
    eps: float = 1e-8
    s_max: float | None = None
    static_s: float = 1.0
    lars_trust: float = 1.0

    def to_c(self) -> _HP:
        s_max = math.sqrt(self.K) if self.s_max is None else self.s_max
        return _HP(self.K, self.rule, self.granularity, self.force_branch,
                   int(bool(self.refresh_scale)), int(bool(self.has_momentum)),
                   self.delta, self.eps, s_max, self.static_s, self.lars_trust)


_lib = None


def _load():
    global _lib
    if _lib is None:
        path = build_oracle()
        lib = ctypes.CDLL(str(path))
        f32p = ctypes.POINTER(ctypes.c_float)
        f64p = ctypes.POINTER(ctypes.c_double)
        pp = ctypes.POINTER(f32p)
        i64p = ctypes.POINTER(ctypes.c_int64)
        lib.oracle_ags_step.argtypes = [pp, pp, pp, i64p, ctypes.c_int, ctypes.c_float,
                                        ctypes.c_float, ctypes.c_float, ctypes.POINTER(_HP),
                                        f32p, pp, f64p, f64p]
        lib.oracle_ags_step.restype = ctypes.c_int
        lib.oracle_ags_step_threads.argtypes = lib.oracle_ags_step.argtypes + [ctypes.c_int]
        lib.oracle_ags_step_threads.restype = ctypes.c_int
        lib.oracle_max_threads.restype = ctypes.c_int
        lib.oracle_layer_stats.argtypes = [pp, pp, ctypes.c_int, i64p, ctypes.c_int, f64p]
        lib.oracle_layer_stats.restype = ctypes.c_int
        lib.oracle_update_scale.argtypes = [pp, pp, i64p, ctypes.c_int, ctypes.c_float,
                                            ctypes.c_float, ctypes.c_int, f32p, pp]
        lib.oracle_update_scale.restype = ctypes.c_int
        lib.oracle_replica_mean.argtypes = [pp, ctypes.c_int, ctypes.c_int64, f32p]
        lib.oracle_sqnorm.argtypes = [f32p, ctypes.c_int64]
        lib.oracle_sqnorm.restype = ctypes.c_double
        lib.oracle_grad_variability.argtypes = [ctypes.c_double, ctypes.c_double, ctypes.c_int64]
        lib.oracle_grad_variability.restype = ctypes.c_double
        lib.oracle_is_scaled.argtypes = [ctypes.c_double, ctypes.c_float, ctypes.c_int]
        lib.oracle_is_scaled.restype = ctypes.c_int
        lib.oracle_scale_tensor.argtypes = [ctypes.c_double, ctypes.c_double, ctypes.c_float,
                                            ctypes.c_float]
        lib.oracle_scale_tensor.restype = ctypes.c_float
        lib.oracle_scale_elementwise.argtypes = [f32p, f32p, ctypes.c_int64, ctypes.c_float,
                                                 ctypes.c_float, f32p]
        _lib = lib
    return _lib


def _f32(a: np.ndarray) -> np.ndarray:
    if a.dtype != np.float32 or not a.flags.c_contiguous or not a.flags.writeable:
        raise TypeError("oracle tensors must be writeable C-contiguous float32 numpy arrays")
    return a


def _fp(a):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_float))


def _ptrs(arrays):
    f32p = ctypes.POINTER(ctypes.c_float)
    arr = (f32p * max(1, len(arrays)))()
    for i, a in enumerate(arrays):
        arr[i] = _fp(_f32(a)) if a is not None else None
    return arr


def replica_mean(grads: list[np.ndarray]) -> np.ndarray:
    """Eq. 1c, fp32, k-ascending sum then division by K."""
    out = np.empty_like(grads[0])
    _load().oracle_replica_mean(_ptrs(grads), len(grads), grads[0].size, _fp(out))
    return out


def sqnorm(x: np.ndarray) -> float:
    """|x|^2 in fp64: exact fp64 squares added from element 0 on with Neumaier's compensated
    summation (within about 1e-16 of the exact sum)."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    return _load().oracle_sqnorm(_fp(x), x.size)


def grad_variability(g2: float, g2_prev: float, steps_done: int) -> float:
    """Eq. 5 (+inf at the first step)."""
    return _load().oracle_grad_variability(g2, g2_prev, steps_done)


def is_scaled(delta_value: float, delta: float, force_branch: int = BRANCH_AUTO) -> bool:
    """Algorithm 1 branch: scaled iff Delta < delta."""
    return bool(_load().oracle_is_scaled(delta_value, delta, force_branch))


def scale_tensor(s_small: float, s_large: float, eps: float, s_max: float) -> float:
    """UpdateGradScale on tensor norms: min(|g_s| / (|g_l| + eps), s_max)."""
    return _load().oracle_scale_tensor(s_small, s_large, eps, s_max)


def scale_elementwise(gs: np.ndarray, gl: np.ndarray, eps: float, s_max: float) -> np.ndarray:
    """UpdateGradScale element-wise: min(|g_s / (g_l + eps)|, s_max)."""
    out = np.empty_like(gs)
    _load().oracle_scale_elementwise(_fp(_f32(gs)), _fp(_f32(gl)), gs.size, eps, s_max, _fp(out))
    return out


def new_state() -> np.ndarray:
    return np.zeros(STATE_LEN, dtype=np.float64)


def max_threads() -> int:
    """Threads ags_step(threads=...) can use (1 when the oracle was built without OpenMP)."""
    return _load().oracle_max_threads()


def ags_step(w, m, grads, lr, momentum, weight_decay, hp: OracleHP, scale=None,
             scale_elem=None, state=None, want_stats=True, threads=None):
    """One optimizer step, in place.  threads: run the per-tensor parts on that many threads
    (the CPU baseline on all host cores); the result is the same bit for bit.

    w, m: lists of n float32 arrays (m may be None when hp.has_momentum is False).
    grads: K lists of n float32 arrays (replica k, tensor p); replica 0 receives
    the mean when K > 1.  scale: float32 [n] (per-tensor gradscale).
    scale_elem: list of n float32 arrays (per-element gradscale).
    state: float64 [4], updated.  Returns the [n, 8] statistics array.
    """
    n = len(w)
    K = hp.K
    assert len(grads) == K and all(len(r) == n for r in grads)
    numel = np.array([a.size for a in w], dtype=np.int64)
    flat_g = [grads[k][p] for k in range(K) for p in range(n)]
    if state is None:
        state = new_state()
    stats = np.zeros((n, STATS_LEN), dtype=np.float64) if want_stats else None
    chp = hp.to_c()
    m_list = m if (m is not None and hp.has_momentum) else [None] * n
    args = (_ptrs(w), _ptrs(m_list), _ptrs(flat_g),
            numel.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)), n, lr, momentum, weight_decay,
            ctypes.byref(chp), _fp(_f32(scale)) if scale is not None else None,
            _ptrs(scale_elem) if scale_elem is not None else None,
            state.ctypes.data_as(ctypes.POINTER(ctypes.c_double)),
            stats.ctypes.data_as(ctypes.POINTER(ctypes.c_double)) if stats is not None else None)
    if threads is None:
        rc = _load().oracle_ags_step(*args)
    else:
        rc = _load().oracle_ags_step_threads(*args, int(threads))
    if rc != 0:
        raise MemoryError("oracle_ags_step failed")
    return stats


def layer_stats(w, grads):
    """Per-layer statistics (no update); replica buffers are left unchanged."""
    n = len(w)
    K = len(grads)
    numel = np.array([a.size for a in w], dtype=np.int64)
    flat_g = [grads[k][p] for k in range(K) for p in range(n)]
    stats = np.zeros((n, STATS_LEN), dtype=np.float64)
    rc = _load().oracle_layer_stats(_ptrs(w), _ptrs(flat_g),
                                    K, numel.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)), n,
                                    stats.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
    if rc != 0:
        raise MemoryError("oracle_layer_stats failed")
    return stats


def update_scale(g_small, g_large, eps, s_max, granularity=GRAN_TENSOR, scale=None,
                 scale_elem=None):
    """UpdateGradScale over tensors: writes scale[p] or scale_elem[p][:]."""
    n = len(g_small)
    numel = np.array([a.size for a in g_small], dtype=np.int64)
    _load().oracle_update_scale(_ptrs(g_small), _ptrs(g_large),
                                numel.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)), n, eps, s_max,
                                granularity, _fp(_f32(scale)) if scale is not None else None,
                                _ptrs(scale_elem) if scale_elem is not None else None)
