"""Shared machinery of the GPU parity tests: one workload held twice, on the
device (driven through the C ABI) and on the host (driven through the oracle),
fed the same seeded inputs, compared after every call.

Tolerances (stated by the task for this method; fp32 data):
  updated w, m:      |gpu - ref| <= 2e-6 |ref| + 1e-7
  per-layer norms:   relative 1e-5
  replica mean:      bitwise (same fp32 operations in the same order)
"""
import math

import numpy as np
import torch

import oracle as O
from paper_2603_18112_gb300 import tula_ags as T
from paper_2603_18112_gb300 import workloads as W

RTOL_W, ATOL_W = 2e-6, 1e-7
RTOL_NORM = 1e-5


def assert_f32_close(gpu, ref, what, rtol=RTOL_W, atol=ATOL_W):
    gpu = np.asarray(gpu, dtype=np.float64).reshape(-1)
    ref = np.asarray(ref, dtype=np.float64).reshape(-1)
    assert gpu.shape == ref.shape, what
    diff = np.abs(gpu - ref)
    bad = ~(diff <= rtol * np.abs(ref) + atol)
    if bad.any():
        i = int(np.argmax(np.where(bad, diff, -1)))
        raise AssertionError(f"{what}: {int(bad.sum())}/{bad.size} outside tolerance; "
                             f"worst at {i}: gpu={gpu[i]!r} ref={ref[i]!r}")


def assert_norm_close(gpu, ref, what, rtol=RTOL_NORM):
    gpu = np.asarray(gpu, dtype=np.float64).reshape(-1)
    ref = np.asarray(ref, dtype=np.float64).reshape(-1)
    both_nan = np.isnan(gpu) & np.isnan(ref)
    ok = both_nan | (np.abs(gpu - ref) <= rtol * np.abs(ref)) | (gpu == ref)
    if not ok.all():
        i = int(np.argmax(~ok))
        raise AssertionError(f"{what}: {int((~ok).sum())} outside rel {rtol}; "
                             f"first at {i}: gpu={gpu[i]!r} ref={ref[i]!r}")


def assert_state_close(gpu, ref, what="state"):
    gpu = np.asarray(gpu, dtype=np.float64)
    assert_norm_close(gpu[0:1], ref[0:1], what + " |G|^2")
    assert gpu[1] == ref[1], what + " steps"
    d_g, d_r = gpu[2], ref[2]
    if math.isinf(d_r) or math.isnan(d_r):
        assert (math.isinf(d_g) and math.isinf(d_r)) or (math.isnan(d_g) and math.isnan(d_r)), \
            f"{what} Delta gpu={d_g} ref={d_r}"
    else:
        assert abs(d_g - d_r) <= 2 * RTOL_NORM * (1 + abs(d_r)), f"{what} Delta {d_g} vs {d_r}"
    assert gpu[3] == ref[3], f"{what} branch gpu={gpu[3]} ref={ref[3]} (Delta {d_g} / {d_r})"


def assert_stats_close(gpu, ref, what="stats"):
    gpu = np.asarray(gpu)
    for c in range(T.TULA_STATS_LEN):
        assert_norm_close(gpu[:, c], ref[:, c], f"{what} col {c}")


class Pair:
    """One workload on the device and on the host."""

    def __init__(self, wl, K=None, align=64, shift=0, with_momentum=True, pset=None,
                 rule=T.TULA_RULE_AGS, granularity=T.TULA_SCALE_PER_TENSOR,
                 force_branch=T.TULA_BRANCH_AUTO, static_s=1.0, lars_trust=1.0, stats=True,
                 grid_ctas=0, s_max=None):
        self.wl = wl
        self.K = wl.K if K is None else K
        self.with_momentum = with_momentum
        self.buf = W.allocate(wl, "cuda", self.K, align, shift, with_momentum, pset)
        W.fill_state(self.buf, wl)
        self.n = self.buf.pset.n_tensors
        self.w_h = W.to_numpy(self.buf.w)
        self.m_h = W.to_numpy(self.buf.m) if with_momentum else None
        self.s_max = (wl.smax if K is None else math.sqrt(self.K)) if s_max is None else s_max
        self.scale_elem = None
        self.scale_elem_h = None
        if granularity == T.TULA_SCALE_PER_ELEMENT:
            gen = torch.Generator(device="cuda")
            gen.manual_seed(wl.seed * 7919 + 5)
            self.scale_elem = [torch.rand(t.shape, generator=gen, device="cuda") * 2.0
                               for t in self.buf.w]
            self.scale_elem_h = W.to_numpy(self.scale_elem)
        self.gpu = T.AGSOptimizerStep(
            self.buf.w, self.buf.g, self.buf.m if with_momentum else None, rule=rule,
            granularity=granularity, s_max=self.s_max, static_s=static_s, lars_trust=lars_trust,
            force_branch=force_branch, scale_elem=self.scale_elem, stats=stats,
            grid_ctas=grid_ctas)
        self.hp = O.OracleHP(K=self.K, rule=rule, granularity=granularity,
                             force_branch=force_branch, has_momentum=with_momentum,
                             s_max=self.s_max, static_s=static_s, lars_trust=lars_trust)
        self.state_h = O.new_state()
        self.scale_h = np.ones(self.n, np.float32)
        self.stats = stats
        self.flags = []

    @property
    def momentum(self):
        return self.wl.momentum if self.with_momentum else 0.0

    def refresh_from(self, g_small_flat):
        """UpdateGradScale (per tensor) with an explicit g_small, replica 0 as g_large."""
        views = W._views(g_small_flat, self.buf.offsets, self.buf.pset.shapes, self.buf.numels)
        hp = T.tula_ags_default_hparams(1)
        hp.s_max = self.s_max
        hp.scale = self.gpu.scale.data_ptr()
        hp.workspace = self.gpu.workspace.data_ptr()
        hp.workspace_bytes = self.gpu.workspace.numel()
        T.tula_ags_update_scale(views, self.buf.g[0], hp)
        O.update_scale(W.to_numpy(views), W.to_numpy(self.buf.g[0]), self.hp.eps, self.s_max,
                       O.GRAN_TENSOR, scale=self.scale_h)
        torch.cuda.synchronize()
        assert_norm_close(self.gpu.scale.cpu().numpy(), self.scale_h, "refreshed scale")

    def step(self, step, mult=1.0, refresh=False, compare=True):
        W.fill_grads(self.buf, self.wl, step, mult)
        g_h = [W.to_numpy(self.buf.g[k]) for k in range(self.K)]
        self.gpu.step(self.wl.lr, self.momentum, self.wl.weight_decay, refresh_scale=refresh)
        self.hp.refresh_scale = refresh
        stats_h = O.ags_step(self.w_h, self.m_h, g_h, self.wl.lr, self.momentum,
                             self.wl.weight_decay, self.hp, scale=self.scale_h,
                             scale_elem=self.scale_elem_h, state=self.state_h)
        torch.cuda.synchronize()
        state = self.gpu.state.cpu().numpy()
        self.flags.append(int(state[3]))
        if not compare:
            return
        where = f"{self.wl.name} K={self.K} step {step}"
        assert_state_close(state, self.state_h, where + " state")
        for p in range(self.n):
            if self.K > 1:
                got = self.buf.g[0][p].reshape(-1).cpu().numpy()
                assert np.array_equal(got, g_h[0][p]), f"{where}: mean of tensor {p}"
            assert_f32_close(self.buf.w[p].reshape(-1).cpu().numpy(), self.w_h[p], f"{where} w[{p}]")
            if self.with_momentum:
                assert_f32_close(self.buf.m[p].reshape(-1).cpu().numpy(), self.m_h[p],
                                 f"{where} m[{p}]")
        if self.stats:
            assert_stats_close(self.gpu.stats.cpu().numpy(), stats_h, where + " stats")
        assert_norm_close(self.gpu.scale.cpu().numpy(), self.scale_h, where + " scale")
