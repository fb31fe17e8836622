"""ctypes binding of libtula_ags (include/tula_ags.h): argument marshalling only.

Every step of the optimizer runs in the CUDA library; this module turns torch
tensors into the C ABI's host pointer arrays and raises on a non-zero status.
It fails loudly (``LibraryNotBuilt``) when the library has not been built --
there is no CPU fallback.  torch is used for device memory and streams only.
"""
from __future__ import annotations

import ctypes
import math
import re
from pathlib import Path

import torch

from .build import HEADER, LIB

c_int, c_float, c_void_p, c_size_t = ctypes.c_int, ctypes.c_float, ctypes.c_void_p, ctypes.c_size_t

TULA_OK, TULA_ERR_ARG, TULA_ERR_WORKSPACE, TULA_ERR_CUDA, TULA_ERR_UNSUPPORTED = 0, -1, -2, -3, -4
TULA_ERR_SCRATCH_LIMIT, TULA_ERR_NO_MEMORY = -5, -6
TULA_STATIC_SCRATCH_BYTES = 16 << 20
TULA_MAX_K = 16
TULA_RULE_AGS, TULA_RULE_NONE, TULA_RULE_LARS, TULA_RULE_STATIC = 0, 1, 2, 3
TULA_SCALE_PER_TENSOR, TULA_SCALE_PER_ELEMENT = 0, 1
TULA_BRANCH_AUTO, TULA_BRANCH_SCALED, TULA_BRANCH_UNSCALED = 0, 1, 2
TULA_STATE_LEN, TULA_STATS_LEN = 4, 8
TULA_G2_SHARE_WORDS = 24
(TULA_STAT_W_SQ, TULA_STAT_G_SQ, TULA_STAT_G0_SQ, TULA_STAT_W_NORM, TULA_STAT_G_NORM,
 TULA_STAT_RATIO, TULA_STAT_COEF, TULA_STAT_SCALE) = range(8)


class LibraryNotBuilt(RuntimeError):
    pass


class TulaError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        msg = tula_ags_error_string(code)
        if code == TULA_ERR_CUDA:
            msg += f" (cudaError {tula_ags_last_cuda_error()})"
        super().__init__(f"{where}: {msg} [{code}]")


class tula_ags_hparams(ctypes.Structure):
    """Mirror of the C struct tula_ags_hparams."""
    _fields_ = [
        ("K", c_int), ("rule", c_int), ("granularity", c_int), ("force_branch", c_int),
        ("refresh_scale", c_int),
        ("delta", c_float), ("eps", c_float), ("s_max", c_float), ("static_s", c_float),
        ("lars_trust", c_float),
        ("scale", c_void_p), ("scale_elem", c_void_p), ("state", c_void_p),
        ("layer_stats", c_void_p), ("workspace", c_void_p), ("workspace_bytes", c_size_t),
        ("grid_ctas", c_int), ("trace_events", c_void_p * 5),
    ]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded library (raises LibraryNotBuilt if it is missing)."""
    global _lib
    if _lib is not None:
        return _lib
    if not LIB.exists():
        raise LibraryNotBuilt(f"{LIB} is missing: run paper_2603_18112_gb300.build.build() "
                              "(or __graft_entry__.build()) first")
    L = ctypes.CDLL(str(LIB))
    pp = ctypes.POINTER(c_void_p)
    i64p = ctypes.POINTER(ctypes.c_int64)
    hpp = ctypes.POINTER(tula_ags_hparams)
    L.tula_ags_default_hparams.argtypes = [hpp, c_int]
    L.tula_ags_default_hparams.restype = None
    L.tula_ags_workspace_size.argtypes = [i64p, c_int, c_int, ctypes.POINTER(c_size_t)]
    L.tula_ags_step.argtypes = [pp, pp, pp, i64p, c_int, c_float, c_float, c_float, hpp, c_void_p]
    L.tula_layer_stats.argtypes = [pp, pp, c_int, i64p, c_int, c_void_p, c_void_p, c_size_t,
                                   c_void_p]
    L.tula_ags_update_scale.argtypes = [pp, pp, i64p, c_int, hpp, c_void_p]
    L.tula_ags_step_static_scratch.argtypes = [pp, pp, pp, i64p, c_int, c_float, c_float,
                                               c_float, hpp, c_void_p]
    L.tula_ags_error_string.argtypes = [c_int]
    L.tula_ags_error_string.restype = ctypes.c_char_p
    L.tula_ags_last_cuda_error.restype = c_int
    L.tula_ags_launch_count.restype = ctypes.c_uint64
    L.tula_ags_plan_chunks.argtypes = [i64p, c_int, c_int, i64p]
    L.tula_ags_chunk_elems.argtypes = [c_int, c_int]
    L.tula_ags_chunk_elems.restype = c_int
    L.tula_ags_workspace_error.argtypes = [c_void_p, c_size_t, i64p, c_int, c_int,
                                           ctypes.POINTER(c_int)]
    L.tula_ags_check_wait_timeout.argtypes = [c_void_p, c_size_t, c_void_p]
    L.tula_ags_static_scratch_error.argtypes = [c_void_p, ctypes.POINTER(c_int)]
    L.tula_ags_shard_reduce.argtypes = [pp, pp, pp, i64p, c_int, c_float, hpp, c_void_p, c_void_p]
    L.tula_ags_shard_update.argtypes = [pp, pp, pp, i64p, c_int, c_float, c_float, c_float, hpp,
                                        c_void_p, c_void_p]
    L.tula_ags_static_scratch_check_wait_timeout.argtypes = [c_void_p]
    L.tula_ags_plan_create.argtypes = [pp, pp, pp, i64p, c_int, hpp, ctypes.POINTER(c_void_p)]
    L.tula_ags_plan_step.argtypes = [c_void_p, c_float, c_float, c_float, hpp, c_void_p]
    L.tula_ags_plan_destroy.argtypes = [c_void_p]
    for name in ("tula_ags_workspace_size", "tula_ags_step", "tula_layer_stats",
                 "tula_ags_update_scale", "tula_ags_plan_chunks", "tula_ags_step_static_scratch",
                 "tula_ags_workspace_error", "tula_ags_check_wait_timeout",
                 "tula_ags_static_scratch_error", "tula_ags_static_scratch_check_wait_timeout",
                 "tula_ags_shard_reduce", "tula_ags_shard_update", "tula_ags_plan_create",
                 "tula_ags_plan_step", "tula_ags_plan_destroy"):
        getattr(L, name).restype = c_int
    _lib = L
    return L


def header_functions() -> list[str]:
    """Names of the functions include/tula_ags.h declares."""
    text = Path(HEADER).read_text()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(tula_\w+)\s*\(", text)) - {"tula_ags_hparams"})


# ---------------------------------------------------------------------------
# marshalling helpers
# ---------------------------------------------------------------------------

def _ptr_array(ptrs):
    arr = (c_void_p * max(1, len(ptrs)))()
    for i, p in enumerate(ptrs):
        arr[i] = p or None
    return arr


def _tensor_ptrs(tensors):
    out = []
    for t in tensors:
        if t is None:
            out.append(None)
            continue
        if t.dtype != torch.float32 or not t.is_contiguous():
            raise TypeError("tensors must be contiguous float32")
        out.append(t.data_ptr())
    return _ptr_array(out)


def _numels(tensors):
    return (ctypes.c_int64 * max(1, len(tensors)))(*[t.numel() for t in tensors])


def _stream_ptr(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _check(rc, where):
    if rc != TULA_OK:
        raise TulaError(rc, where)


def _replica_list(params, grads, hp, where, moms=None):
    """grads[k][p] flattened k-major, after checking that it holds hp.K replicas of every
    tensor (and one momentum buffer per tensor): the library reads K * n gradient pointers and
    n momentum pointers, so a shorter list must not reach it."""
    n = len(params)
    if moms is not None and len(moms) != n:
        raise ValueError(f"{where}: {len(moms)} momentum buffers for {n} tensors")
    if hp is not None and hp.K != len(grads):
        raise ValueError(f"{where}: hp.K = {hp.K} but {len(grads)} replica lists were given")
    for k, r in enumerate(grads):
        if len(r) != n:
            raise ValueError(f"{where}: replica {k} has {len(r)} tensors, params has {n}")
    return [grads[k][p] for k in range(len(grads)) for p in range(n)]


# ---------------------------------------------------------------------------
# C-ABI functions, same names
# ---------------------------------------------------------------------------

def tula_ags_error_string(code: int) -> str:
    return lib().tula_ags_error_string(code).decode()


def tula_ags_last_cuda_error() -> int:
    return lib().tula_ags_last_cuda_error()


def tula_ags_launch_count() -> int:
    return lib().tula_ags_launch_count()


def tula_ags_chunk_elems(pass_: int, streams: int) -> int:
    """Elements per tile of pass 1 (reduction) or pass 2 (update) with `streams` streams."""
    return lib().tula_ags_chunk_elems(pass_, streams)


def tula_ags_check_wait_timeout(workspace: torch.Tensor, stream=None) -> None:
    """Launches the bounded-wait check (about a second on the GPU): afterwards the workspace's
    error word has bit 0 set, as after a stage that never filled."""
    _check(lib().tula_ags_check_wait_timeout(c_void_p(workspace.data_ptr()),
                                             workspace.numel() * workspace.element_size(),
                                             _stream_ptr(stream)),
           "tula_ags_check_wait_timeout")


def tula_ags_workspace_error(workspace: torch.Tensor, numels, K: int) -> int:
    """Reads and clears the workspace's error word (synchronous): 0 = every wait completed."""
    arr = (ctypes.c_int64 * max(1, len(numels)))(*[int(n) for n in numels])
    out = c_int(0)
    _check(lib().tula_ags_workspace_error(c_void_p(workspace.data_ptr()),
                                          workspace.numel() * workspace.element_size(), arr,
                                          len(numels), K, ctypes.byref(out)),
           "tula_ags_workspace_error")
    return out.value


def tula_ags_default_hparams(K: int) -> tula_ags_hparams:
    hp = tula_ags_hparams()
    lib().tula_ags_default_hparams(ctypes.byref(hp), K)
    return hp


def tula_ags_workspace_size(numels, K: int = 1) -> int:
    arr = (ctypes.c_int64 * max(1, len(numels)))(*[int(n) for n in numels])
    out = c_size_t(0)
    _check(lib().tula_ags_workspace_size(arr, len(numels), K, ctypes.byref(out)),
           "tula_ags_workspace_size")
    return out.value


def tula_ags_plan_chunks(numels, chunk_elems: int) -> list[int]:
    arr = (ctypes.c_int64 * max(1, len(numels)))(*[int(n) for n in numels])
    out = (ctypes.c_int64 * (len(numels) + 1))()
    _check(lib().tula_ags_plan_chunks(arr, len(numels), chunk_elems, out), "tula_ags_plan_chunks")
    return list(out)


def new_workspace(numels, K: int = 1, device="cuda") -> torch.Tensor:
    """A zero-filled, 256-byte aligned workspace tensor (torch allocations are)."""
    n = tula_ags_workspace_size(numels, K)
    return torch.zeros(n, dtype=torch.uint8, device=device)


def tula_ags_step(params, grads, moms, lr, momentum, weight_decay, hp: tula_ags_hparams,
                  stream=None, _cache=None) -> None:
    """One optimizer step.  params, moms: lists of n tensors (moms may be None);
    grads: K lists of n tensors (grads[k][p]); hp: tula_ags_hparams."""
    n = len(params)
    flat = _replica_list(params, grads, hp, "tula_ags_step", moms)
    rc = lib().tula_ags_step(_tensor_ptrs(params), _tensor_ptrs(flat),
                             _tensor_ptrs(moms) if moms is not None else None, _numels(params), n,
                             lr, momentum, weight_decay, ctypes.byref(hp), _stream_ptr(stream))
    _check(rc, "tula_ags_step")


def tula_ags_plan_create(params, grads, moms, hp: tula_ags_hparams) -> c_void_p:
    """A plan over fixed tensors (hp.K, hp.scale_elem read); the tensors must outlive it."""
    flat = _replica_list(params, grads, hp, "tula_ags_plan_create", moms)
    plan = c_void_p()
    rc = lib().tula_ags_plan_create(_tensor_ptrs(params), _tensor_ptrs(flat),
                                    _tensor_ptrs(moms) if moms is not None else None,
                                    _numels(params), len(params), ctypes.byref(hp),
                                    ctypes.byref(plan))
    _check(rc, "tula_ags_plan_create")
    return plan


def tula_ags_plan_step(plan: c_void_p, lr, momentum, weight_decay, hp: tula_ags_hparams,
                       stream=None) -> None:
    rc = lib().tula_ags_plan_step(plan, lr, momentum, weight_decay, ctypes.byref(hp),
                                  _stream_ptr(stream))
    _check(rc, "tula_ags_plan_step")


def tula_ags_plan_destroy(plan: c_void_p) -> None:
    _check(lib().tula_ags_plan_destroy(plan), "tula_ags_plan_destroy")


def tula_ags_step_static_scratch(params, grads, moms, lr, momentum, weight_decay,
                                 hp: tula_ags_hparams, stream=None) -> None:
    """tula_ags_step for callers that cannot allocate device memory: the step's scratch is
    the library's static device array (hp.workspace is ignored).  Calls on one device must not
    overlap on the GPU; make the first call on a device before any stream capture."""
    n = len(params)
    flat = _replica_list(params, grads, hp, "tula_ags_step_static_scratch", moms)
    rc = lib().tula_ags_step_static_scratch(
        _tensor_ptrs(params), _tensor_ptrs(flat), _tensor_ptrs(moms) if moms is not None else None,
        _numels(params), n, lr, momentum, weight_decay, ctypes.byref(hp), _stream_ptr(stream))
    _check(rc, "tula_ags_step_static_scratch")


def tula_ags_static_scratch_error(stream=None) -> int:
    """Reads and clears the static scratch's error word after the work on `stream`
    (synchronous): 0 = every wait of the static-scratch steps since the last read completed."""
    out = c_int(0)
    _check(lib().tula_ags_static_scratch_error(_stream_ptr(stream), ctypes.byref(out)),
           "tula_ags_static_scratch_error")
    return out.value


def tula_ags_static_scratch_check_wait_timeout(stream=None) -> None:
    """The bounded-wait check against the static scratch's error word (about two seconds on
    the GPU): afterwards tula_ags_static_scratch_error reports bit 0."""
    _check(lib().tula_ags_static_scratch_check_wait_timeout(_stream_ptr(stream)),
           "tula_ags_static_scratch_check_wait_timeout")


def tula_layer_stats(params, grads, stats_out: torch.Tensor, workspace: torch.Tensor,
                     stream=None) -> None:
    n = len(params)
    K = len(grads)
    flat = _replica_list(params, grads, None, "tula_layer_stats")
    rc = lib().tula_layer_stats(_tensor_ptrs(params), _tensor_ptrs(flat), K, _numels(params), n,
                                c_void_p(stats_out.data_ptr()), c_void_p(workspace.data_ptr()),
                                workspace.numel() * workspace.element_size(), _stream_ptr(stream))
    _check(rc, "tula_layer_stats")


def tula_ags_update_scale(g_small, g_large, hp: tula_ags_hparams, stream=None) -> None:
    n = len(g_small)
    if len(g_large) != n:
        raise ValueError(f"tula_ags_update_scale: {n} small-batch and {len(g_large)} "
                         "large-batch tensors")
    rc = lib().tula_ags_update_scale(_tensor_ptrs(g_small), _tensor_ptrs(g_large),
                                     _numels(g_small), n, ctypes.byref(hp), _stream_ptr(stream))
    _check(rc, "tula_ags_update_scale")


# ---------------------------------------------------------------------------
# Pre-marshalled step for a fixed set of tensors (what a training loop calls)
# ---------------------------------------------------------------------------

class AGSOptimizerStep:
    """Holds the pointer arrays, state, scale, statistics and workspace of one
    model so that each step is a single C call.

    params, moms: n tensors; grads: K lists of n tensors (replica k of tensor p).
    plan: step through a tula_ags_plan (sizes and pointers checked once, launch tables
    reused) rather than through tula_ags_step; the results are the same bit for bit.
    """

    def __init__(self, params, grads, moms=None, *, rule=TULA_RULE_AGS,
                 granularity=TULA_SCALE_PER_TENSOR, delta=0.5, eps=1e-8, s_max=None,
                 static_s=1.0, lars_trust=1.0, force_branch=TULA_BRANCH_AUTO, scale=None,
                 scale_elem=None, stats=True, grid_ctas=0, plan=True):
        self.params = list(params)
        self.grads = [list(r) for r in grads]
        self.moms = list(moms) if moms is not None else None
        self.n = len(self.params)
        self.K = len(self.grads)
        if not 1 <= self.K <= TULA_MAX_K:
            raise ValueError(f"AGSOptimizerStep: {self.K} replica lists (1 .. {TULA_MAX_K})")
        if self.moms is not None and len(self.moms) != self.n:
            raise ValueError(f"AGSOptimizerStep: {len(self.moms)} momentum buffers for "
                             f"{self.n} tensors")
        dev = self.params[0].device
        self.hp = tula_ags_default_hparams(self.K)
        self.hp.rule = rule
        self.hp.granularity = granularity
        self.hp.delta = delta
        self.hp.eps = eps
        self.hp.s_max = math.sqrt(self.K) if s_max is None else s_max
        self.hp.static_s = static_s
        self.hp.lars_trust = lars_trust
        self.hp.force_branch = force_branch
        self.hp.grid_ctas = grid_ctas
        self.state = torch.zeros(TULA_STATE_LEN, dtype=torch.float64, device=dev)
        self.scale = (scale if scale is not None else
                      torch.ones(self.n, dtype=torch.float32, device=dev))
        self.stats = (torch.zeros(self.n, TULA_STATS_LEN, dtype=torch.float64, device=dev)
                      if stats else None)
        self.workspace = new_workspace([t.numel() for t in self.params], self.K, dev)
        self.hp.scale = self.scale.data_ptr()
        self.hp.state = self.state.data_ptr()
        self.hp.layer_stats = self.stats.data_ptr() if self.stats is not None else None
        self.hp.workspace = self.workspace.data_ptr()
        self.hp.workspace_bytes = self.workspace.numel()
        self._scale_elem = None
        if scale_elem is not None:
            self._scale_elem_tensors = list(scale_elem)
            self._scale_elem = _tensor_ptrs(self._scale_elem_tensors)
            self.hp.scale_elem = ctypes.cast(self._scale_elem, c_void_p).value
        flat = _replica_list(self.params, self.grads, self.hp, "AGSOptimizerStep")
        self._p = _tensor_ptrs(self.params)
        self._g = _tensor_ptrs(flat)
        self._m = _tensor_ptrs(self.moms) if self.moms is not None else None
        self._numels = _numels(self.params)
        self._plan = None
        if plan:
            handle = c_void_p()
            _check(lib().tula_ags_plan_create(self._p, self._g, self._m, self._numels, self.n,
                                              ctypes.byref(self.hp), ctypes.byref(handle)),
                   "tula_ags_plan_create")
            self._plan = handle
            self._destroy = lib().tula_ags_plan_destroy  # kept for __del__ at shutdown
        # The zero fills above ran on the current stream; steps may be issued on any other
        # (torch's side streams do not wait for it), so finish them before the first step.
        torch.cuda.synchronize(dev)

    def set_trace_events(self, events):
        """Up to five cudaEvent_t handles (or None) recorded at the kernel boundaries of a
        step: before the reduction, after it, after its combine, after the update, after the
        update's combine."""
        for i in range(5):
            ev = events[i] if events is not None and i < len(events) else None
            self.hp.trace_events[i] = (ev.cuda_event if hasattr(ev, "cuda_event") else ev) or None

    def error(self) -> int:
        """Reads and clears the workspace error word (synchronous); 0 = all waits completed."""
        return tula_ags_workspace_error(self.workspace, [t.numel() for t in self.params], self.K)

    def step(self, lr, momentum, weight_decay, refresh_scale=False, stream=None) -> None:
        self.hp.refresh_scale = 1 if refresh_scale else 0
        if self._plan is not None:
            rc = lib().tula_ags_plan_step(self._plan, lr, momentum, weight_decay,
                                          ctypes.byref(self.hp), _stream_ptr(stream))
            _check(rc, "tula_ags_plan_step")
            return
        rc = lib().tula_ags_step(self._p, self._g, self._m, self._numels, self.n, lr, momentum,
                                 weight_decay, ctypes.byref(self.hp), _stream_ptr(stream))
        _check(rc, "tula_ags_step")

    def __del__(self):
        plan = getattr(self, "_plan", None)
        if plan is not None:
            self._plan = None
            self._destroy(plan)

    __call__ = step

    # -- a step sharded over ranks: this object holds one rank's tensors --------------------

    def new_g2_share(self) -> torch.Tensor:
        """A device buffer for a share of |G|^2 (TULA_G2_SHARE_WORDS uint64, held as int64: the
        integer sums of the exchange wrap the same way)."""
        return torch.zeros(TULA_G2_SHARE_WORDS, dtype=torch.int64, device=self.params[0].device)

    def shard_reduce(self, momentum, g2_share: torch.Tensor, refresh_scale=False,
                     stream=None) -> None:
        """Pass 1 on this rank's tensors; its share of |G|^2 into g2_share."""
        self.hp.refresh_scale = 1 if refresh_scale else 0
        rc = lib().tula_ags_shard_reduce(self._p, self._g, self._m, self._numels, self.n, momentum,
                                         ctypes.byref(self.hp), c_void_p(g2_share.data_ptr()),
                                         _stream_ptr(stream))
        _check(rc, "tula_ags_shard_reduce")

    def shard_update(self, lr, momentum, weight_decay, g2_total: torch.Tensor,
                     refresh_scale=False, stream=None) -> None:
        """The rest of the step on this rank's tensors, from every rank's share summed."""
        self.hp.refresh_scale = 1 if refresh_scale else 0
        rc = lib().tula_ags_shard_update(self._p, self._g, self._m, self._numels, self.n, lr,
                                         momentum, weight_decay, ctypes.byref(self.hp),
                                         c_void_p(g2_total.data_ptr()), _stream_ptr(stream))
        _check(rc, "tula_ags_shard_update")


def combine_g2_shares(share: torch.Tensor, group=None) -> torch.Tensor:
    """The exchange of a sharded step: every rank's share of |G|^2 summed, in place, over the
    torch.distributed group (an integer SUM, exact and independent of the reduction order).
    Without an initialised process group or with one rank, the share is the total."""
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized() and dist.get_world_size(group) > 1:
        dist.all_reduce(share, op=dist.ReduceOp.SUM, group=group)
    return share


def sharded_step(step: AGSOptimizerStep, lr, momentum, weight_decay, group=None,
                 refresh_scale=False, share=None) -> torch.Tensor:
    """One step sharded over the group's ranks: shard_reduce, the exchange, shard_update, all
    on the current stream.  Returns the summed share."""
    share = step.new_g2_share() if share is None else share
    step.shard_reduce(momentum, share, refresh_scale)
    combine_g2_shares(share, group)
    step.shard_update(lr, momentum, weight_decay, share, refresh_scale)
    return share
