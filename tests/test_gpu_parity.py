"""GPU parity: the CUDA library (through its C ABI) against the CPU oracle on the
same seeded inputs, element by element, over multi-step runs that take both
branches of Algorithm 1, at sizes that span many chunks and ragged tails and at
the full sizes of the paper's parameter sets."""
import math

import numpy as np
import pytest
import torch

import oracle as O
from _parity import (Pair, assert_f32_close, assert_norm_close, assert_state_close,
                     assert_stats_close)
from paper_2603_18112_gb300 import tula_ags as T
from paper_2603_18112_gb300 import workloads as W

pytestmark = pytest.mark.gpu

CHUNK = 16384  # an arbitrary ragged boundary; the tile sizes themselves come from the library


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2603_18112_gb300 import build
    build.build()
    T.lib()


def _ragged_pset(extra=(), K=None):
    """Empty, tiny and ragged tensors; with K, also sizes one below, at and one above a tile and
    two tiles of every pass (the tile sizes the library uses for K replicas: pass 1, pass 2, and
    pass 1 reading w)."""
    ps = W.ParamSet("ragged")
    sizes = [0, 1, 3, 4, 5, 63, 64, 65, 4095, CHUNK - 1, CHUNK, CHUNK + 1, 40000, 100003, *extra]
    if K is not None:
        for t in (T.tula_ags_chunk_elems(1, K), T.tula_ags_chunk_elems(2, 3),
                  T.tula_ags_chunk_elems(3, K + 1)):
            sizes += [t - 1, t, t + 1, 2 * t + 1]
    for n in sizes:
        ps.add((n,), W.KIND_NORMAL)
    return ps


def test_resnet20_ten_steps():
    """ResNet-20 parameter set, K = 1, the 10-step multiplier schedule (both branches)."""
    wl = W.workload("resnet20")
    pair = Pair(wl)
    W.fill_grads(pair.buf, wl, step=0)
    small = torch.empty_like(pair.buf.g_flats[0])
    W.fill_small(pair.buf, wl, small, step=0)
    pair.refresh_from(small)
    for i, mult in enumerate(W.STEP_MULTIPLIERS):
        pair.step(i + 1, mult)
    assert pair.flags[0] == 0 and 1 in pair.flags and pair.flags[3] == 0  # x2 jump: sensitive


@pytest.mark.parametrize("K", [1, 2, 3, 4, 5, 8, 16])
@pytest.mark.parametrize("shift", [0, 1])
@pytest.mark.parametrize("rule", [T.TULA_RULE_AGS, T.TULA_RULE_LARS])
def test_ragged_shapes(K, shift, rule):
    """Tensors of 0..100003 elements (ragged chunk tails); shift=1 misaligns every tensor.  LARS
    takes pass 1 through its own ring (w read), K = 3 and 5 through the kernel compiled for any
    K."""
    wl = W.workload("stress_k4", seed=11 + K, factor_range=(1e-3, 1e1), zero_patterns=False)
    pair = Pair(wl, K=K, align=1 if shift else 64, shift=shift, pset=_ragged_pset(K=K), rule=rule,
                lars_trust=0.01)
    # draw 1 twice (Delta = 0: scaled), then x2 (Delta = 3: unscaled), then a fresh draw
    for i, (seed_step, mult) in enumerate(((1, 1.0), (1, 1.0), (1, 2.0), (2, 1.0))):
        pair.step(seed_step, mult, refresh=(K > 1 and i == 0))
    assert pair.flags[:3] == [0, 1, 0]


@pytest.mark.parametrize("name", ["resnet18", "resnet50", "vgg16"])
def test_full_parameter_sets(name):
    """Full-size ResNet-18 (K=4), ResNet-50 (K=8), VGG-16 (K=8): refresh, scaled, unscaled."""
    wl = W.workload(name)
    pair = Pair(wl)
    for i, mult in enumerate((1.0, 1.0, 2.0)):
        pair.step(1, mult, refresh=(i == 0))
    assert pair.flags == [0, 1, 0]


@pytest.mark.parametrize("rule,gran,mom", [
    (T.TULA_RULE_NONE, T.TULA_SCALE_PER_TENSOR, True),
    (T.TULA_RULE_LARS, T.TULA_SCALE_PER_TENSOR, True),
    (T.TULA_RULE_STATIC, T.TULA_SCALE_PER_TENSOR, True),
    (T.TULA_RULE_AGS, T.TULA_SCALE_PER_ELEMENT, True),
    (T.TULA_RULE_AGS, T.TULA_SCALE_PER_TENSOR, False),
])
def test_rules(rule, gran, mom):
    wl = W.workload("resnet20", seed=21)
    pair = Pair(wl, K=2, rule=rule, granularity=gran, with_momentum=mom, static_s=4.0,
                lars_trust=0.01, s_max=2.0)
    for i, (seed_step, mult) in enumerate(((1, 1.0), (1, 1.0), (1, 2.0), (2, 1.0))):
        pair.step(seed_step, mult, refresh=(gran == T.TULA_SCALE_PER_TENSOR and i == 0))
    assert pair.flags[:3] == [0, 1, 0]


@pytest.mark.parametrize("rule", [T.TULA_RULE_AGS, T.TULA_RULE_LARS])
def test_many_tensors_span_several_launches(rule):
    """1000 tensors with K = 16 need several parameter blocks per pass (LARS: pass 1 reading w,
    through its own ring and tile size)."""
    rng = np.random.default_rng(5)
    ps = W.ParamSet("many")
    for n in rng.integers(1, 5000, size=1000):
        ps.add((int(n),), W.KIND_NORMAL)
    wl = W.workload("stress_k16", seed=31)
    pair = Pair(wl, pset=ps, rule=rule, lars_trust=0.01)
    before = T.tula_ags_launch_count()
    for i, mult in enumerate((1.0, 1.0)):
        pair.step(i + 1, mult, refresh=(i == 0))
    assert T.tula_ags_launch_count() - before >= 2 * 2 * 2


def test_zero_gradients_and_weights():
    """All-zero gradients: |G|^2 = 0, the next step has Delta = inf/NaN -> unscaled."""
    ps = _ragged_pset()
    wl = W.workload("stress_k4", seed=41, factor_range=(0.0, 0.0))
    wl = W.Workload(**{**wl.__dict__, "factor_range": None, "grad_std": 0.0, "w_std": 0.0})
    pair = Pair(wl, K=4, pset=ps, rule=T.TULA_RULE_LARS)
    pair.step(1, 1.0)
    pair.step(2, 1.0)
    st = pair.gpu.state.cpu().numpy()
    assert st[0] == 0.0 and st[3] == 0.0
    assert np.all(pair.gpu.stats.cpu().numpy()[:, T.TULA_STAT_COEF] == 1.0)


def _inputs_snapshot(buf):
    return ([f.clone() for f in buf.g_flats], buf.w_flat.clone(),
            buf.m_flat.clone() if buf.m_flat is not None else None)


def _restore(buf, snap):
    for f, s in zip(buf.g_flats, snap[0]):
        f.copy_(s)
    buf.w_flat.copy_(snap[1])
    if snap[2] is not None:
        buf.m_flat.copy_(snap[2])


@pytest.mark.parametrize("name", ["resnet18", "resnet50"])
def test_bitwise_reproducible_across_runs_and_grids(name):
    wl = W.workload(name)
    buf = W.allocate(wl, "cuda")
    W.fill_state(buf, wl)
    W.fill_grads(buf, wl, step=1)
    snap = _inputs_snapshot(buf)
    outs = []
    for grid in (0, 0, 1, 7, 333):
        _restore(buf, snap)
        st = T.AGSOptimizerStep(buf.w, buf.g, buf.m, grid_ctas=grid)
        st.state.copy_(torch.tensor([1.0, 3.0, 0.0, 0.0], dtype=torch.float64))
        st.step(wl.lr, wl.momentum, wl.weight_decay, refresh_scale=True)
        st.step(wl.lr, wl.momentum, wl.weight_decay)  # and a step without refresh
        torch.cuda.synchronize()
        outs.append([buf.g_flats[0].clone(), buf.w_flat.clone(), buf.m_flat.clone(),
                     st.stats.clone(), st.state.clone(), st.scale.clone()])
    for o in outs[1:]:
        for a, b in zip(outs[0], o):
            assert torch.equal(a, b)


@pytest.mark.parametrize("K", [1, 3, 4])
def test_layer_stats(K):
    wl = W.workload("resnet18", seed=51)
    buf = W.allocate(wl, "cuda", K=K)
    W.fill_state(buf, wl)
    W.fill_grads(buf, wl, step=1)
    g_before = [f.clone() for f in buf.g_flats]
    ws = T.new_workspace(buf.numels, K)
    stats = torch.zeros(buf.pset.n_tensors, 8, dtype=torch.float64, device="cuda")
    T.tula_layer_stats(buf.w, buf.g, stats, ws)
    ref = O.layer_stats(W.to_numpy(buf.w), [W.to_numpy(buf.g[k]) for k in range(K)])
    torch.cuda.synchronize()
    assert_stats_close(stats.cpu().numpy(), ref, "layer_stats")
    for a, b in zip(g_before, buf.g_flats):
        assert torch.equal(a, b)  # read-only


@pytest.mark.parametrize("gran", [T.TULA_SCALE_PER_TENSOR, T.TULA_SCALE_PER_ELEMENT])
def test_update_scale(gran):
    wl = W.workload("resnet20", seed=61)
    buf = W.allocate(wl, "cuda", K=2, pset=_ragged_pset(extra=(7, 300001)))
    W.fill_grads(buf, wl, step=1)
    gs, gl = buf.g[0], buf.g[1]
    hp = T.tula_ags_default_hparams(4)
    hp.granularity = gran
    n = buf.pset.n_tensors
    scale = torch.zeros(n, dtype=torch.float32, device="cuda")
    ws = T.new_workspace(buf.numels, 1)
    hp.scale, hp.workspace, hp.workspace_bytes = scale.data_ptr(), ws.data_ptr(), ws.numel()
    se = [torch.zeros_like(t) for t in gs]
    keep = None
    if gran == T.TULA_SCALE_PER_ELEMENT:
        keep = T._tensor_ptrs(se)
        hp.scale_elem = T.ctypes.cast(keep, T.c_void_p).value
    T.tula_ags_update_scale(gs, gl, hp)
    ref_scale = np.zeros(n, np.float32)
    ref_se = [np.zeros(t.numel(), np.float32) for t in gs]
    O.update_scale(W.to_numpy(gs), W.to_numpy(gl), 1e-8, 2.0, gran, scale=ref_scale,
                   scale_elem=ref_se)
    torch.cuda.synchronize()
    if gran == T.TULA_SCALE_PER_TENSOR:
        assert_norm_close(scale.cpu().numpy(), ref_scale, "scale")
    else:
        for p in range(n):
            assert np.array_equal(se[p].reshape(-1).cpu().numpy(), ref_se[p]), p


def _oracle_g2(buf, K):
    """|G|^2 of the replica mean over every tensor, one tensor at a time (oracle)."""
    total = 0.0
    for p in range(buf.pset.n_tensors):
        g = [buf.g[k][p].reshape(-1).cpu().numpy() for k in range(K)]
        total += O.sqnorm(O.replica_mean(g))
    return total


def test_steps_replayed_from_a_cuda_graph():
    """A captured step (no allocation, no host synchronisation, kernels chained by programmatic
    dependent launch) replays to the same bytes as the same steps issued one by one."""
    wl = W.workload("resnet18")
    bufs, steps = [], []
    for _ in range(2):
        buf = W.allocate(wl, "cuda")
        W.fill_state(buf, wl)
        W.fill_grads(buf, wl, step=1)
        bufs.append(buf)
        steps.append(T.AGSOptimizerStep(buf.w, buf.g, buf.m, s_max=wl.smax))
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        for st in steps:  # one eager step each: the library sets itself up outside capture
            st.step(wl.lr, wl.momentum, wl.weight_decay, refresh_scale=True, stream=s)
    s.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        steps[1].step(wl.lr, wl.momentum, wl.weight_decay, stream=s)
    for i in range(4):
        with torch.cuda.stream(s):
            steps[0].step(wl.lr, wl.momentum, wl.weight_decay, stream=s)
            g.replay()
        s.synchronize()
        a, b = bufs
        assert torch.equal(a.w_flat, b.w_flat) and torch.equal(a.m_flat, b.m_flat), i
        assert torch.equal(a.g_flats[0], b.g_flats[0]), i
        assert torch.equal(steps[0].state, steps[1].state), i
        assert torch.equal(steps[0].stats, steps[1].stats), i
    assert steps[0].state[1].item() == 5.0  # five steps taken: the refresh step and four more


def test_a_tensor_past_2_31_elements():
    """One tensor of 2.6e9 elements (K = 2; element indices past 2^31), constant per role so
    that every element has the same closed-form result, which the oracle gives on a few
    elements: sampled elements around 2^31 and at both ends, the extremes over the whole
    tensor, and |G|^2 = n |gbar|^2."""
    K = 2
    n = 1_694_208 * min(T.tula_ags_chunk_elems(1, K + 1), T.tula_ags_chunk_elems(2, 4))
    assert n > 2 ** 31
    need = (K + 2) * 4 * n + (1 << 30)
    if torch.cuda.mem_get_info()[0] < need:
        pytest.skip(f"needs {need / 1e9:.0f} GB of device memory")
    vals = {"w": 0.5, "m": 0.01, "g0": 0.003, "g1": -0.001}
    w = torch.full((n,), vals["w"], device="cuda")
    m = torch.full((n,), vals["m"], device="cuda")
    g = [torch.full((n,), vals["g0"], device="cuda"), torch.full((n,), vals["g1"], device="cuda")]
    st = T.AGSOptimizerStep([w], [[g[0]], [g[1]]], [m])
    lr, mu, wd = 0.1, 0.9, 5e-4
    st.step(lr, mu, wd)
    torch.cuda.synchronize()

    # the oracle on four elements of the same values
    w_h = [np.full(4, vals["w"], np.float32)]
    m_h = [np.full(4, vals["m"], np.float32)]
    g_h = [[np.full(4, vals["g0"], np.float32)], [np.full(4, vals["g1"], np.float32)]]
    state_h = O.new_state()
    O.ags_step(w_h, m_h, g_h, lr, mu, wd, O.OracleHP(K=K), scale=np.ones(1, np.float32),
               state=state_h)
    idx = torch.tensor([0, 1, 2 ** 31 - 1, 2 ** 31, 2 ** 31 + 1, n // 2, n - 2, n - 1],
                       device="cuda")
    for got, want, what in ((w, w_h[0][0], "w"), (m, m_h[0][0], "m"), (g[0], g_h[0][0][0], "mean")):
        assert torch.all(got[idx] == float(want)), what
        assert got.min().item() == float(want) and got.max().item() == float(want), what
    gbar = float(g_h[0][0][0])
    g2 = st.state[0].item()
    assert g2 == pytest.approx(n * gbar * gbar, rel=1e-5)
    assert st.stats[0, T.TULA_STAT_G_SQ].item() == pytest.approx(n * gbar * gbar, rel=1e-5)
    assert st.state[3].item() == 0.0  # the first step is unscaled


@pytest.mark.parametrize("name", ["stress_k1", "stress_k4", "stress_k16"])
def test_stress_full_size_sampled(name):
    """The ~1.65e9-element stress set at full size, in the benchmark's launch shape: |G|^2
    against the oracle over every tensor; w, m, mean and statistics on 160 sampled tensors
    (including the all-zero patterns and the largest tensor); a forced scaled second step."""
    wl = W.workload(name)
    K = wl.K
    buf = W.allocate(wl, "cuda")
    W.fill_state(buf, wl)
    n = buf.pset.n_tensors
    numels = buf.numels
    rng = np.random.default_rng(9)
    sample = sorted(set(rng.choice(n, 150, replace=False).tolist())
                    | {7, 13, 21, 64 + 7, int(np.argmax(numels)), int(np.argmin(numels))})
    gpu = T.AGSOptimizerStep(buf.w, buf.g, buf.m, s_max=wl.smax)
    hp = O.OracleHP(K=K, s_max=wl.smax)
    w_h = [buf.w[p].reshape(-1).cpu().numpy().copy() for p in sample]
    m_h = [buf.m[p].reshape(-1).cpu().numpy().copy() for p in sample]
    scale_h = np.ones(len(sample), np.float32)
    if K == 1:
        W.fill_grads(buf, wl, step=0)
        small = torch.empty_like(buf.g_flats[0])
        W.fill_small(buf, wl, small, step=0)
        views = W._views(small, buf.offsets, buf.pset.shapes, numels)
        T.tula_ags_update_scale(views, buf.g[0], gpu.hp)
        O.update_scale([views[p].reshape(-1).cpu().numpy() for p in sample],
                       [buf.g[0][p].reshape(-1).cpu().numpy() for p in sample], hp.eps,
                       wl.smax, O.GRAN_TENSOR, scale=scale_h)
        del small, views
    for step, force in ((1, O.BRANCH_AUTO), (2, O.BRANCH_SCALED)):
        W.fill_grads(buf, wl, step=step)
        g_h = [[buf.g[k][p].reshape(-1).cpu().numpy().copy() for p in sample] for k in range(K)]
        g2 = _oracle_g2(buf, K) if step == 1 else None
        gpu.hp.force_branch = force
        gpu.step(wl.lr, wl.momentum, wl.weight_decay, refresh_scale=(K > 1 and step == 1))
        hp.force_branch = force if step == 2 else O.BRANCH_AUTO
        hp.refresh_scale = K > 1 and step == 1
        st_h = O.new_state()
        stats_h = O.ags_step(w_h, m_h, g_h, wl.lr, wl.momentum, wl.weight_decay, hp,
                             scale=scale_h, state=st_h)
        torch.cuda.synchronize()
        state = gpu.state.cpu().numpy()
        stats = gpu.stats.cpu().numpy()
        if step == 1:
            assert_state_close(state, np.array([g2, 1.0, math.inf, 0.0]), name)
            g2_prev = state[0]
        else:
            assert state[3] == 1.0
            assert state[2] == pytest.approx(abs((state[0] - g2_prev) / g2_prev), rel=1e-12)
            # |G|^2 is the fixed-order sum of the per-layer |gbar|^2
            assert state[0] == pytest.approx(float(np.sum(stats[:, T.TULA_STAT_G_SQ])), rel=1e-12)
        for i, p in enumerate(sample):
            where = f"{name} step {step} tensor {p}"
            if K > 1:
                assert np.array_equal(buf.g[0][p].reshape(-1).cpu().numpy(), g_h[0][i]), where
            assert_f32_close(buf.w[p].reshape(-1).cpu().numpy(), w_h[i], where + " w")
            assert_f32_close(buf.m[p].reshape(-1).cpu().numpy(), m_h[i], where + " m")
            for c in (0, 1, 2, 3, 4, 5, 6, 7):
                assert_norm_close(stats[p, c:c + 1], stats_h[i, c:c + 1], f"{where} stat {c}")
        assert_norm_close(gpu.scale.cpu().numpy()[sample], scale_h, name + " scale")
    del buf, gpu
    torch.cuda.empty_cache()


def test_a_wait_that_runs_out_is_reported_and_the_context_survives():
    """Failure detection without a fault: the library's bounded mbarrier wait, on a barrier
    nothing arrives on, gives up (about a second), sets the workspace's error word, and the
    next step on the same context runs and matches the oracle."""
    import time
    wl = W.workload("resnet20")
    pair = Pair(wl)
    numels = [t.numel() for t in pair.buf.w]
    ws = pair.gpu.workspace
    assert T.tula_ags_workspace_error(ws, numels, pair.K) == 0
    t0 = time.perf_counter()
    T.tula_ags_check_wait_timeout(ws)
    torch.cuda.synchronize()
    waited = time.perf_counter() - t0
    assert T.tula_ags_workspace_error(ws, numels, pair.K) == 1  # reported, then cleared
    assert T.tula_ags_workspace_error(ws, numels, pair.K) == 0
    assert 0.05 < waited < 60.0
    pair.step(1, 1.0)  # the context is still usable and the step still exact
    assert T.tula_ags_workspace_error(ws, numels, pair.K) == 0


@pytest.mark.parametrize("K", [1, 4])
def test_calls_back_to_back_on_one_workspace_and_stream(K):
    """A step, tula_layer_stats, a step, tula_ags_update_scale and a step issued on one stream
    and one workspace with no synchronisation between them (a step's first kernels start before
    the call ahead of them has completed) give what the oracle gives for the same sequence."""
    wl = W.workload("stress_k4", seed=71 + K, factor_range=(1e-2, 1e1), zero_patterns=False)
    pair = Pair(wl, K=K, pset=_ragged_pset(K=K))
    buf, gpu = pair.buf, pair.gpu
    W.fill_grads(buf, wl, step=1)
    g_h = [W.to_numpy(buf.g[k]) for k in range(K)]
    small = torch.empty_like(buf.g_flats[0])
    W.fill_small(buf, wl, small, step=1)
    small_views = W._views(small, buf.offsets, buf.pset.shapes, buf.numels)
    small_h = W.to_numpy(small_views)
    stats_mid = torch.zeros(pair.n, T.TULA_STATS_LEN, dtype=torch.float64, device="cuda")
    hp = T.tula_ags_default_hparams(1)
    hp.s_max = pair.s_max
    hp.scale = gpu.scale.data_ptr()
    hp.workspace, hp.workspace_bytes = gpu.workspace.data_ptr(), gpu.workspace.numel()
    lr, mu, wd = wl.lr, pair.momentum, wl.weight_decay
    torch.cuda.synchronize()
    gpu.step(lr, mu, wd)
    T.tula_layer_stats(buf.w, buf.g, stats_mid, gpu.workspace)
    gpu.step(lr, mu, wd)
    T.tula_ags_update_scale(small_views, buf.g[0], hp)
    gpu.step(lr, mu, wd)
    torch.cuda.synchronize()

    def oracle_step():
        return O.ags_step(pair.w_h, pair.m_h, g_h, lr, mu, wd, pair.hp, scale=pair.scale_h,
                          state=pair.state_h)

    oracle_step()
    stats_mid_h = O.layer_stats(pair.w_h, g_h)
    oracle_step()
    O.update_scale(small_h, g_h[0], pair.hp.eps, pair.s_max, O.GRAN_TENSOR, scale=pair.scale_h)
    stats_h = oracle_step()

    assert_stats_close(stats_mid.cpu().numpy(), stats_mid_h, "layer_stats between steps")
    assert_norm_close(gpu.scale.cpu().numpy(), pair.scale_h, "scale refreshed between steps")
    assert_state_close(gpu.state.cpu().numpy(), pair.state_h, "state after three steps")
    assert_stats_close(gpu.stats.cpu().numpy(), stats_h, "stats of the third step")
    for p in range(pair.n):
        assert np.array_equal(buf.g[0][p].reshape(-1).cpu().numpy(), g_h[0][p]), p
        assert_f32_close(buf.w[p].reshape(-1).cpu().numpy(), pair.w_h[p], f"w[{p}]")
        assert_f32_close(buf.m[p].reshape(-1).cpu().numpy(), pair.m_h[p], f"m[{p}]")


def _extreme_pset(*tiles):
    """Tensors of one element to several tiles (ragged tails) of each pass-1 tile given as
    (pass, streams) -- pass 3 is pass 1 when it reads w -- three times over, for per-tensor
    gradient factors spread over 46 decades."""
    ps = W.ParamSet("extremes")
    for pass_, streams in tiles:
        t = T.tula_ags_chunk_elems(pass_, streams)
        for _ in range(3):
            for n in (1, 5, 64, 1000, t - 1, t + 3, 2 * t + 7, 40000):
                ps.add((n,), W.KIND_NORMAL)
    return ps


def _extreme_workload(seed, ps):
    wl = W.workload("stress_k4", seed=seed, factor_range=(1e-24, 1e22), zero_patterns=False)
    f = W._factors(wl, ps)
    # squares below fp32's normal range, beyond its largest value, and ordinary ones
    assert (f < 1e-20).any() and (f > 1e20).any() and ((f > 1e-3) & (f < 1e3)).any()
    return wl


def test_lars_steps_over_the_whole_float_range():
    """LARS steps take every pass-1 norm precisely.  Gradient factors from 1e-24 to 1e22: the
    squares of some tensors underflow or overflow fp32 (they go through fp64), the others are
    split exactly into float-float pairs; coefficients, norms and updates match the oracle."""
    ps = _extreme_pset((3, 3))
    wl = _extreme_workload(97, ps)
    pair = Pair(wl, K=2, pset=ps, rule=T.TULA_RULE_LARS, lars_trust=0.01)
    pair.step(1, 1.0)
    pair.step(2, 1.0)


def test_update_scale_over_the_whole_float_range():
    """UpdateGradScale per tensor (precise norms of g_small and g_large) over the same range,
    with s_max out of the way: each scale within 2 ulp of the oracle's fp64 ratio."""
    ps = _extreme_pset((1, 2))
    wl = _extreme_workload(105, ps)
    buf = W.allocate(wl, "cuda", K=2, pset=ps)
    W.fill_grads(buf, wl, step=1)
    gs, gl = buf.g[1], buf.g[0]
    n = buf.pset.n_tensors
    hp = T.tula_ags_default_hparams(2)
    hp.s_max = 1e30
    scale = torch.zeros(n, dtype=torch.float32, device="cuda")
    ws = T.new_workspace(buf.numels, 1)
    hp.scale, hp.workspace, hp.workspace_bytes = scale.data_ptr(), ws.data_ptr(), ws.numel()
    T.tula_ags_update_scale(gs, gl, hp)
    ref = np.zeros(n, np.float32)
    O.update_scale(W.to_numpy(gs), W.to_numpy(gl), hp.eps, 1e30, O.GRAN_TENSOR, scale=ref)
    torch.cuda.synchronize()
    assert_norm_close(scale.cpu().numpy(), ref, "scale", rtol=2.0 ** -22)


def _scale_weights(pair, seed, lo=1e-24, hi=1e22):
    """Multiplies each tensor's w by its own factor, the factors evenly spaced in log from lo to
    hi and shuffled, on both sides (the same fp32 products), so that weight squares underflow,
    overflow and stay ordinary."""
    rng = np.random.default_rng([seed, 9])
    f = np.exp(rng.permutation(np.linspace(math.log(lo), math.log(hi), pair.n))).astype(np.float32)
    assert (f < 1e-20).any() and (f > 1e20).any()
    for p, t in enumerate(pair.buf.w):
        t.mul_(float(f[p]))
    torch.cuda.synchronize()
    pair.w_h = W.to_numpy(pair.buf.w)


def test_default_steps_over_the_whole_float_range():
    """Algorithm 1 steps on the default path (fp32 sums within a tile, no refresh, no LARS) and
    tula_layer_stats, with gradient and weight factors from 1e-24 to 1e22: tiles whose fp32
    sums of squares would overflow, underflow, or hold only zeros are summed again with an exact
    power-of-two scaling; norms, |G|^2, Delta, the branch, w and m match the oracle."""
    ps = _extreme_pset((1, 2), (3, 3))   # the step's pass 1, and tula_layer_stats' (reads w)
    wl = _extreme_workload(113, ps)
    pair = Pair(wl, K=2, pset=ps)
    _scale_weights(pair, 113)
    rng = np.random.default_rng(114)
    s0 = rng.uniform(0.5, 2.0, size=pair.n).astype(np.float32)   # a non-trivial gradscale
    pair.gpu.scale.copy_(torch.from_numpy(s0))
    pair.scale_h = s0.copy()
    # unscaled (first step), scaled (Delta = 0), unscaled (x2: Delta = 3)
    for seed_step, mult in ((1, 1.0), (1, 1.0), (1, 2.0)):
        pair.step(seed_step, mult)
    assert pair.flags == [0, 1, 0]
    # the statistics alone, read-only, over the same range
    W.fill_grads(pair.buf, wl, step=2)
    stats = torch.zeros(pair.n, T.TULA_STATS_LEN, dtype=torch.float64, device="cuda")
    T.tula_layer_stats(pair.buf.w, pair.buf.g, stats, pair.gpu.workspace)
    ref = O.layer_stats(W.to_numpy(pair.buf.w), [W.to_numpy(pair.buf.g[k]) for k in range(2)])
    torch.cuda.synchronize()
    assert_stats_close(stats.cpu().numpy(), ref, "layer_stats over the whole float range")
    big = ref[:, T.TULA_STAT_W_SQ] > 3.4e38
    tiny = (ref[:, T.TULA_STAT_G_SQ] > 0) & (ref[:, T.TULA_STAT_G_SQ] < 1e-38)
    assert big.any() and tiny.any()  # the case is what it claims to be


@pytest.mark.parametrize("K", [1, 4])
def test_default_steps_misaligned_over_the_whole_float_range(K):
    """The same range on misaligned tensors, where every element is loaded one by one (fp64
    squares), and with K = 1 and 4 (other tile sizes and stream counts)."""
    ps = _extreme_pset((1, K if K > 1 else 1))
    wl = _extreme_workload(121 + K, ps)
    for shift in (0, 1):
        pair = Pair(wl, K=K, pset=ps, align=1 if shift else 64, shift=shift)
        _scale_weights(pair, 121 + K)
        pair.step(1, 1.0)
        pair.step(1, 1.0)
        assert pair.flags == [0, 1]


@pytest.mark.parametrize("K", [1, 8])
def test_norms_are_exact_sums_on_integer_data(K):
    """With small integers in every replica and weight, every square and every fp32 tile sum is
    exact, so the exact accumulation across tiles must give the oracle's norms bit for bit (the
    oracle's compensated fp64 sums are exact here too), and |G|^2 must be the exact sum of the
    per-tensor |gbar|^2, for any grid size."""
    ps = _ragged_pset(extra=(3_000_001,), K=K)
    wl = W.workload("stress_k4", seed=131 + K, zero_patterns=False)
    buf = W.allocate(wl, "cuda", K=K, pset=ps)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(131 + K)
    for f in [buf.w_flat] + buf.g_flats:
        f.copy_(torch.randint(-7, 8, f.shape, generator=gen, device="cuda").float())
    ref = O.layer_stats(W.to_numpy(buf.w), [W.to_numpy(buf.g[k]) for k in range(K)])
    cols = (T.TULA_STAT_W_SQ, T.TULA_STAT_G_SQ, T.TULA_STAT_G0_SQ)
    for col in cols:
        assert np.all(ref[:, col] == np.round(ref[:, col] * 64) / 64)  # exact, as claimed
    g2 = float(np.sum(ref[:, T.TULA_STAT_G_SQ]))  # exact: every term a multiple of 1/64
    stats = torch.zeros(buf.pset.n_tensors, 8, dtype=torch.float64, device="cuda")
    T.tula_layer_stats(buf.w, buf.g, stats, T.new_workspace(buf.numels, K))
    torch.cuda.synchronize()
    for col in cols:
        assert np.array_equal(stats.cpu().numpy()[:, col], ref[:, col]), ("layer_stats", col)
    snap = _inputs_snapshot(buf)
    for grid in (0, 1, 13, 333):
        _restore(buf, snap)
        st = T.AGSOptimizerStep(buf.w, buf.g, buf.m, grid_ctas=grid)
        st.step(0.1, 0.9, 0.0)
        torch.cuda.synchronize()
        got = st.stats.cpu().numpy()
        for col in cols:
            assert np.array_equal(got[:, col], ref[:, col]), (grid, col)
        assert st.state[0].item() == g2, grid


@pytest.mark.parametrize("n", [1, 3, 4, 5, 8, 9])
@pytest.mark.parametrize("rule", [T.TULA_RULE_AGS, T.TULA_RULE_LARS])
def test_tensor_counts_around_a_finish_block(n, rule):
    """The finish kernel runs one warp per tensor, four per block, plus one warp for the step
    record: tensor counts that fill whole blocks, and those that do not, both get their record
    (|G|^2, Delta, branch) and every tensor's statistics, in the step that takes the branch in
    the update (AGS) and in the one with a finish between the passes (LARS)."""
    ps = W.ParamSet("count")
    for i in range(n):
        ps.add((1000 + 517 * i,), W.KIND_NORMAL)
    wl = W.workload("stress_k4", seed=141 + n, factor_range=(0.1, 10.0), zero_patterns=False)
    pair = Pair(wl, K=2, pset=ps, rule=rule, lars_trust=0.01)
    for seed_step, mult in ((1, 1.0), (1, 1.0), (1, 2.0)):
        pair.step(seed_step, mult)
    assert pair.flags == [0, 1, 0]


def test_checkpoint_and_resume_through_the_host():
    """All AGS state lives in caller buffers (w, m, the gradscale, the step record), so a
    checkpoint is a copy of them: 3 steps, the state copied to the host, a fresh optimizer step
    (new device buffers, new workspace) built from those copies, 3 more steps -- bitwise the
    same as 6 uninterrupted steps, statistics included, across both branches and a refresh."""
    wl = W.workload("stress_k4", seed=151, factor_range=(0.1, 10.0), zero_patterns=False)
    ps = _ragged_pset(K=4)
    schedule = [(1, 1.0, True), (2, 1.0, False), (2, 1.0, False), (3, 2.0, False),
                (4, 1.0, True), (4, 1.0, False)]

    def fresh():
        buf = W.allocate(wl, "cuda", K=4, pset=ps)
        W.fill_state(buf, wl)
        return buf

    def run(buf, st, steps):
        for seed_step, mult, refresh in steps:
            W.fill_grads(buf, wl, step=seed_step, multiplier=mult)
            st.step(wl.lr, wl.momentum, wl.weight_decay, refresh_scale=refresh)
        torch.cuda.synchronize()

    a = fresh()
    st_a = T.AGSOptimizerStep(a.w, a.g, a.m, s_max=2.0)
    run(a, st_a, schedule)

    b = fresh()
    st_b = T.AGSOptimizerStep(b.w, b.g, b.m, s_max=2.0)
    run(b, st_b, schedule[:3])
    ckpt = {"w": b.w_flat.cpu().numpy().copy(), "m": b.m_flat.cpu().numpy().copy(),
            "state": st_b.state.cpu().numpy().copy(), "scale": st_b.scale.cpu().numpy().copy()}
    del st_b, b
    torch.cuda.empty_cache()

    c = fresh()  # new buffers: the same shapes, contents replaced from the checkpoint
    c.w_flat.copy_(torch.from_numpy(ckpt["w"]))
    c.m_flat.copy_(torch.from_numpy(ckpt["m"]))
    st_c = T.AGSOptimizerStep(c.w, c.g, c.m, s_max=2.0,
                              scale=torch.from_numpy(ckpt["scale"]).cuda())
    st_c.state.copy_(torch.from_numpy(ckpt["state"]))
    torch.cuda.synchronize()
    run(c, st_c, schedule[3:])

    assert [int(x) for x in (st_a.state[3].item(), st_c.state[3].item())] == [1, 1]
    assert st_a.state[1].item() == st_c.state[1].item() == 6.0
    for x, y in ((a.w_flat, c.w_flat), (a.m_flat, c.m_flat), (a.g_flats[0], c.g_flats[0]),
                 (st_a.state, st_c.state), (st_a.scale, st_c.scale), (st_a.stats, st_c.stats)):
        assert torch.equal(x, y)


@pytest.mark.parametrize("name,rule", [("resnet50", T.TULA_RULE_AGS), ("resnet18", T.TULA_RULE_LARS),
                                       ("ragged_k4", T.TULA_RULE_AGS)])
def test_sharded_step_equals_the_whole_step(name, rule):
    """A step sharded over two ranks (each owning whole tensors) run on one GPU, one shard after
    the other: each rank's pass 1 exports its share of |G|^2, the shares are summed as integers,
    and each rank finishes from the sum.  Tiles are cut per tensor and the sums are exact, so the
    mean, every norm, |G|^2, Delta, the branch, w, m and the gradscale equal those of one step
    over all tensors bit for bit -- whichever order the shares are added in."""
    if name == "ragged_k4":
        wl = W.workload("stress_k4", seed=161, factor_range=(0.1, 10.0), zero_patterns=False)
        ps = _ragged_pset(K=4)
    else:
        wl, ps = W.workload(name), None
    K = 4 if ps is not None else wl.K
    a, b = (W.allocate(wl, "cuda", K=K, pset=ps) for _ in range(2))
    for buf in (a, b):
        W.fill_state(buf, wl)
    n = a.pset.n_tensors
    cut = n // 2 + 1
    kw = dict(s_max=2.0, rule=rule, lars_trust=0.01)
    whole = T.AGSOptimizerStep(a.w, a.g, a.m, **kw)
    ranks = [T.AGSOptimizerStep(b.w[lo:hi], [b.g[k][lo:hi] for k in range(K)], b.m[lo:hi], **kw)
             for lo, hi in ((0, cut), (cut, n))]
    shares = [r.new_g2_share() for r in ranks]
    for i, (seed_step, mult) in enumerate(((1, 1.0), (1, 1.0), (1, 2.0), (2, 1.0))):
        refresh = rule == T.TULA_RULE_AGS and i == 0
        for buf in (a, b):
            W.fill_grads(buf, wl, step=seed_step, multiplier=mult)
        whole.step(wl.lr, wl.momentum, wl.weight_decay, refresh_scale=refresh)
        for r, sh in zip(ranks, shares):
            r.shard_reduce(wl.momentum, sh, refresh_scale=refresh)
        total = shares[1] + shares[0] if i % 2 else shares[0] + shares[1]  # either order
        for r in ranks:
            r.shard_update(wl.lr, wl.momentum, wl.weight_decay, total, refresh_scale=refresh)
        torch.cuda.synchronize()
        where = f"{name} step {i + 1}"
        for r in ranks:
            assert torch.equal(r.state, whole.state), where + " state"
        assert torch.equal(torch.cat([r.stats for r in ranks]), whole.stats), where + " stats"
        assert torch.equal(torch.cat([r.scale for r in ranks]), whole.scale), where + " scale"
        for x, y in ((a.w_flat, b.w_flat), (a.m_flat, b.m_flat), (a.g_flats[0], b.g_flats[0])):
            assert torch.equal(x, y), where
    assert [int(v) for v in (whole.state[1].item(),)] == [4]


@pytest.mark.gpu
@pytest.mark.parametrize("case", ["ragged_k4", "many_k2", "no_momentum"])
def test_plan_steps_equal_direct_steps(case):
    """A plan (tula_ags_plan_create) checks the tensors once and keeps the launch tables of each
    kernel variant from its first use.  Switching rule, granularity, refresh, branch and grid
    between steps -- each a variant the plan builds once and then reuses -- must give bit for bit
    the w, m, mean, step record, statistics and gradscale of tula_ags_step with the same
    arguments.  The plan also refuses what it was not created with."""
    if case == "many_k2":
        rng = np.random.default_rng(171)
        ps = W.ParamSet("many")
        for n in rng.integers(1, 3000, size=800):   # several parameter blocks per pass
            ps.add((int(n),), W.KIND_NORMAL)
        K = 2
    else:
        ps, K = _ragged_pset(K=4), 4
    mom = case != "no_momentum"
    wl = W.workload("stress_k4", seed=171, factor_range=(0.1, 10.0), zero_patterns=False)
    bufs = [W.allocate(wl, "cuda", K=K, pset=ps, with_momentum=mom) for _ in range(2)]
    for b in bufs:
        W.fill_state(b, wl)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(172)
    se0 = [torch.rand(t.numel(), generator=gen, device="cuda") * 2 for t in bufs[0].w]
    se = [se0, [x.clone() for x in se0]]
    kw = dict(s_max=2.0, lars_trust=0.01, static_s=0.5)
    st = [T.AGSOptimizerStep(b.w, b.g, b.m if mom else None, scale_elem=se[i], plan=(i == 0), **kw)
          for i, b in enumerate(bufs)]
    assert st[0]._plan is not None and st[1]._plan is None
    mu = 0.9 if mom else 0.0
    schedule = [
        (1, 1.0, dict(refresh=True)),
        (1, 1.0, dict()),                                    # Delta = 0: scaled
        (2, 2.0, dict(grid=7)),                              # Delta = 3: unscaled
        (2, 1.0, dict(rule=T.TULA_RULE_LARS)),
        (3, 1.0, dict(gran=T.TULA_SCALE_PER_ELEMENT, force=T.TULA_BRANCH_SCALED)),
        (3, 1.0, dict(gran=T.TULA_SCALE_PER_ELEMENT)),
        (4, 1.0, dict(rule=T.TULA_RULE_STATIC, force=T.TULA_BRANCH_SCALED, grid=333)),
        (4, 1.0, dict(rule=T.TULA_RULE_NONE)),
        (5, 1.0, dict(refresh=True)),
        (5, 1.0, dict()),
    ]
    for i, (seed_step, mult, o) in enumerate(schedule):
        for b, s in zip(bufs, st):
            W.fill_grads(b, wl, step=seed_step, multiplier=mult)
            s.hp.rule = o.get("rule", T.TULA_RULE_AGS)
            s.hp.granularity = o.get("gran", T.TULA_SCALE_PER_TENSOR)
            s.hp.force_branch = o.get("force", T.TULA_BRANCH_AUTO)
            s.hp.grid_ctas = o.get("grid", 0)
            s.step(wl.lr, mu, wl.weight_decay, refresh_scale=o.get("refresh", False))
        torch.cuda.synchronize()
        where = f"{case} step {i + 1} {o}"
        a, b = bufs
        assert torch.equal(a.w_flat, b.w_flat), where + " w"
        assert torch.equal(a.g_flats[0], b.g_flats[0]), where + " mean"
        if mom:
            assert torch.equal(a.m_flat, b.m_flat), where + " m"
        for name in ("state", "stats", "scale"):   # bit patterns: the statistics hold NaN
            x, y = getattr(st[0], name), getattr(st[1], name)
            it = torch.int64 if x.dtype == torch.float64 else torch.int32
            assert torch.equal(x.view(it), y.view(it)), where + " " + name
    assert st[0].state[1].item() == len(schedule)
    p = st[0]
    p.hp.rule, p.hp.granularity, p.hp.force_branch, p.hp.grid_ctas = T.TULA_RULE_AGS, 0, 0, 0
    p.hp.K = K + 1                                             # not the plan's K
    with pytest.raises(T.TulaError) as e:
        p.step(0.1, mu, 0.0)
    assert e.value.code == T.TULA_ERR_ARG
    p.hp.K = K
    if not mom:
        with pytest.raises(T.TulaError) as e:                  # no momentum buffers in the plan
            p.step(0.1, 0.9, 0.0)
        assert e.value.code == T.TULA_ERR_ARG
    bare = T.AGSOptimizerStep(bufs[0].w, bufs[0].g, bufs[0].m if mom else None, **kw)
    bare.hp.granularity = T.TULA_SCALE_PER_ELEMENT             # created without scale_elem
    with pytest.raises(T.TulaError) as e:
        bare.step(0.1, mu, 0.0)
    assert e.value.code == T.TULA_ERR_ARG
    torch.cuda.synchronize()
    assert p.error() == 0


@pytest.mark.gpu
@pytest.mark.parametrize("delta", [0.5, 0.1, 0.3, 1.0, 0.25, 2.0])
def test_branch_at_the_rounding_boundary_of_delta(delta):
    """Algorithm 1's branch where the rounded Delta of Eq. 5 meets delta.  |G|^2 is fixed by
    integer gradients (K = 1, so the sum is exact); the previous |G|^2 is planted in the step
    record on both sides of G2 and stepped one ulp at a time across the point where
    fl(|fl(G2 - G2_prev)| / G2_prev) reaches delta.  Delta (bit for bit) and the branch must be
    those of the fp64 formula for every candidate, both branches must occur, and a first step
    (no previous norm) is unscaled."""
    n = 4099
    gen = torch.Generator(device="cuda")
    gen.manual_seed(181)
    g = torch.randint(-9, 10, (n,), generator=gen, device="cuda").float()
    g2 = float(np.sum(g.cpu().numpy().astype(np.float64) ** 2))   # exact: integers < 2^53
    w = torch.zeros(n, device="cuda")
    m = torch.zeros(n, device="cuda")
    st = T.AGSOptimizerStep([w], [[g]], [m], s_max=1.0, delta=delta, stats=False)
    d32 = float(np.float32(delta))
    seen = set()
    for sign in (1.0, -1.0):
        if sign < 0 and d32 >= 1.0:
            continue                              # G2_prev would have to be negative
        centre = g2 / (1.0 + sign * d32)          # |g2 - g2p| / g2p = delta near here
        cands = [centre]
        for direction in (np.inf, -np.inf):
            x = centre
            for _ in range(6):
                x = float(np.nextafter(x, direction))
                cands.append(x)
        for g2p in cands:
            st.state.copy_(torch.tensor([g2p, 3.0, 0.0, 0.0], dtype=torch.float64))
            st.step(0.0, 0.0, 0.0)
            torch.cuda.synchronize()
            dv = abs((np.float64(g2) - np.float64(g2p)) / np.float64(g2p))
            want = int(dv < np.float64(d32))
            got = st.state.cpu().numpy()
            assert got[0] == g2 and got[1] == 4.0, g2p
            assert got[2] == dv, (g2p, got[2], dv)
            assert int(got[3]) == want, (delta, g2p, dv)
            seen.add(want)
    assert seen == {0, 1}
    st.state.zero_()                              # a first step: Delta = +inf, unscaled
    st.step(0.0, 0.0, 0.0)
    torch.cuda.synchronize()
    got = st.state.cpu().numpy()
    assert np.isinf(got[2]) and got[3] == 0.0
    assert st.error() == 0
