"""Pins of the CPU oracle to what the paper and the mathematics fix (no GPU).

Each test ties one part of the oracle to something other than itself: a
textbook or library routine (torch.optim.SGD), a closed form, brute force on
tiny inputs, a hand-worked example, an invariant of Lemma 1, or a value the
paper prints (tests/golden/paper_hparams.json).  A dropped term, a wrong sign,
a transposed operand or a wrong index in the oracle fails at least one.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_hparams.json")
U32 = 2.0 ** -24  # unit roundoff of fp32


def _rand(rng, numels, scale=1.0):
    return [(rng.standard_normal(n) * scale).astype(np.float32) for n in numels]


def _close(a, b, rel=2e-6, abs_=1e-7):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return np.all(np.abs(a - b) <= rel * np.abs(b) + abs_)


# --------------------------------------------------------------------------
# Paper-printed values
# --------------------------------------------------------------------------

def test_paper_defaults_golden():
    """delta = 0.5, eps = 1e-8 (Algorithm 1 inputs, Sec. IV-B); s_max = sqrt(b_l / b_s)."""
    gold = json.load(open(GOLDEN))
    hp = O.OracleHP(K=8)
    assert hp.delta == gold["delta"]["value"]
    assert hp.eps == gold["eps"]["value"]
    # b_small = one replica's share of b_large = b_large / K  =>  s_max = sqrt(K)
    assert hp.to_c().s_max == pytest.approx(math.sqrt(8), rel=1e-7)


# --------------------------------------------------------------------------
# Eq. 1c: replica mean
# --------------------------------------------------------------------------

def test_mean_exact_for_representable_inputs():
    a = np.array([1.0, 3.0, -2.5, 0.0, 1e-3], np.float32)
    b = np.array([3.0, 1.0, 0.5, -0.0, 3e-3], np.float32)
    got = O.replica_mean([a, b])
    assert np.array_equal(got[:4], np.array([2.0, 2.0, -1.0, 0.0], np.float32))
    assert got[4] == np.float32((np.float32(1e-3) + np.float32(3e-3)) / np.float32(2))


@pytest.mark.parametrize("K", [1, 2, 3, 4, 5, 8, 16])
def test_mean_brute_force_fp64(K):
    rng = np.random.default_rng(K)
    g = _rand(rng, [257] * K)
    got = O.replica_mean(g).astype(np.float64)
    exact = np.sum(np.stack([x.astype(np.float64) for x in g]), axis=0) / K
    mag = np.sum(np.abs(np.stack(g).astype(np.float64)), axis=0) / K
    # K-1 fp32 additions and one division: |err| <= K * u * (sum |g_k|) / K
    assert np.all(np.abs(got - exact) <= (K + 1) * U32 * mag + 1e-30)
    # each replica counted with weight 1/K: dropping one moves the mean by |g_k|/K
    if K > 1:
        dropped = np.sum(np.stack(g[1:]).astype(np.float64), axis=0) / K
        assert not np.allclose(got, dropped)


def test_mean_order_is_k_ascending():
    # fp32: (1e8 + 4) rounds to a multiple of 8, so ((g0 + g1) + g2) != g1, while the
    # association (g0 + g2) + g1 would give exactly 4: the result shows the order used
    a = np.array([1e8], np.float32)
    b = np.array([4.0], np.float32)
    c = np.array([-1e8], np.float32)
    got = O.replica_mean([a, b, c])
    expect = np.float32(np.float32(np.float32(a[0] + b[0]) + c[0]) / np.float32(3))
    assert got[0] == expect
    assert got[0] != np.float32(4.0 / 3.0)  # the order matters here, and it is k = 0, 1, 2


# --------------------------------------------------------------------------
# Norms (|G|^2 of Eq. 5, per-layer statistics)
# --------------------------------------------------------------------------

@pytest.mark.parametrize("n", [0, 1, 3, 5, 64, 65, 1000])
def test_sqnorm_brute_force(n):
    rng = np.random.default_rng(n)
    x = (rng.standard_normal(n) * 10.0 ** rng.uniform(-6, 6, n)).astype(np.float32)
    exact = math.fsum(float(v) * float(v) for v in x)  # squares exact in fp64; fsum exact
    got = O.sqnorm(x)
    # compensated summation: within ~2 fp64 roundings of the exact sum, independent of n
    assert abs(got - exact) <= 4 * 2.0 ** -53 * exact + 0.0


def test_sqnorm_accuracy_independent_of_length():
    rng = np.random.default_rng(99)
    x = (rng.standard_normal(2_000_000) * 10.0 ** rng.uniform(-3, 3, 2_000_000)).astype(np.float32)
    xs = x.astype(np.float64)
    exact = math.fsum((xs * xs).tolist())
    assert abs(O.sqnorm(x) - exact) <= 4 * 2.0 ** -53 * exact


def test_sqnorm_closed_forms():
    assert O.sqnorm(np.ones(1000, np.float32)) == 1000.0
    assert O.sqnorm(np.full(77, 0.5, np.float32)) == 77 * 0.25
    assert O.sqnorm(np.full(3, -3.0, np.float32)) == 27.0
    assert O.sqnorm(np.zeros(5, np.float32)) == 0.0


# --------------------------------------------------------------------------
# Eq. 5 and the branch of Algorithm 1, through full steps
# --------------------------------------------------------------------------

def _one_tensor_step(g_list, state, hp, w=None, scale=None):
    n = g_list[0].size
    w = [np.zeros(n, np.float32) if w is None else w]
    m = [np.zeros(n, np.float32)]
    grads = [[g.copy()] for g in g_list]
    stats = O.ags_step(w, m, grads, 0.1, 0.9, 0.0, hp, scale=scale, state=state)
    return w[0], m[0], stats


@pytest.mark.parametrize("mults,expect", [
    ((1.0, 2.0), 3.0),      # |G|^2 x4:   |(4 - 1) / 1| = 3
    ((2.0, 1.0), 0.75),     # |G|^2 / 4:  |(1/4 - 1)| = 0.75
    ((1.0, 1.0), 0.0),
    ((4.0, 1.0), 15.0 / 16.0),
])
def test_delta_closed_forms(mults, expect):
    rng = np.random.default_rng(1)
    base = rng.standard_normal(100).astype(np.float32)
    hp = O.OracleHP(K=1)
    state = O.new_state()
    _one_tensor_step([base * np.float32(mults[0])], state, hp, scale=np.ones(1, np.float32))
    assert state[1] == 1 and math.isinf(state[2]) and state[3] == 0  # first step: sensitive
    _one_tensor_step([base * np.float32(mults[1])], state, hp, scale=np.ones(1, np.float32))
    assert state[1] == 2
    assert state[2] == pytest.approx(expect, abs=1e-12)
    assert state[3] == (1.0 if expect < 0.5 else 0.0)


def test_delta_small_change():
    rng = np.random.default_rng(2)
    base = rng.standard_normal(1000).astype(np.float32)
    hp = O.OracleHP(K=1)
    state = O.new_state()
    _one_tensor_step([base], state, hp, scale=np.ones(1, np.float32))
    _one_tensor_step([base * np.float32(1.1)], state, hp, scale=np.ones(1, np.float32))
    assert state[2] == pytest.approx(0.21, rel=1e-6)  # 1.1^2 - 1
    assert state[3] == 1.0


def test_branch_is_strict_at_threshold():
    # |G_prev|^2 = 2, |G|^2 = 3  =>  Delta = 0.5 exactly = delta  =>  unscaled (Delta >= delta)
    hp = O.OracleHP(K=1, delta=0.5)
    state = O.new_state()
    _one_tensor_step([np.array([1, 1, 0], np.float32)], state, hp, scale=np.ones(1, np.float32))
    _one_tensor_step([np.array([1, 1, 1], np.float32)], state, hp, scale=np.ones(1, np.float32))
    assert state[2] == 0.5 and state[3] == 0.0
    assert O.is_scaled(0.49999999, 0.5) and not O.is_scaled(0.5, 0.5)
    assert not O.is_scaled(float("nan"), 0.5) and not O.is_scaled(float("inf"), 0.5)
    assert O.is_scaled(9.0, 0.5, O.BRANCH_SCALED) and not O.is_scaled(0.0, 0.5, O.BRANCH_UNSCALED)


def test_zero_previous_norm_is_sensitive():
    hp = O.OracleHP(K=1)
    state = O.new_state()
    _one_tensor_step([np.zeros(4, np.float32)], state, hp, scale=np.ones(1, np.float32))
    _one_tensor_step([np.ones(4, np.float32)], state, hp, scale=np.ones(1, np.float32))
    assert math.isinf(state[2]) and state[3] == 0.0
    assert O.grad_variability(0.0, 0.0, 3) != O.grad_variability(0.0, 0.0, 3)  # NaN
    assert math.isinf(O.grad_variability(1.0, 5.0, 0))


# --------------------------------------------------------------------------
# The update: unscaled = textbook momentum SGD; Algorithm 1's update line
# --------------------------------------------------------------------------

@pytest.mark.parametrize("rule,force", [(O.RULE_NONE, O.BRANCH_AUTO),
                                        (O.RULE_AGS, O.BRANCH_UNSCALED),
                                        (O.RULE_STATIC, O.BRANCH_UNSCALED)])
def test_unscaled_step_is_torch_sgd(rule, force):
    """c = 1 reduces the step to torch.optim.SGD(momentum, weight_decay) on the mean gradient."""
    rng = np.random.default_rng(3)
    numels = [1, 7, 33, 130, 1025]
    K = 2
    lr, mu, wd = 0.1, 0.9, 5e-4
    w = _rand(rng, numels)
    m = [np.zeros(n, np.float32) for n in numels]
    tw = [torch.nn.Parameter(torch.from_numpy(a.copy())) for a in w]
    opt = torch.optim.SGD(tw, lr=lr, momentum=mu, weight_decay=wd, dampening=0.0, nesterov=False,
                          foreach=False)
    hp = O.OracleHP(K=K, rule=rule, force_branch=force, static_s=8.0)
    scale = rng.uniform(0.2, 3.0, len(numels)).astype(np.float32)
    state = O.new_state()
    for step in range(6):
        g = [_rand(rng, numels, 1e-2) for _ in range(K)]
        for p, t in enumerate(tw):
            t.grad = torch.stack([torch.from_numpy(g[k][p].copy()) for k in range(K)]).mean(0)
        O.ags_step(w, m, g, lr, mu, wd, hp, scale=scale, state=state)
        opt.step()
        for p, t in enumerate(tw):
            assert _close(w[p], t.detach().numpy()), (step, p)
            assert _close(m[p], opt.state[t]["momentum_buffer"].numpy()), (step, p)


@pytest.mark.parametrize("force", [O.BRANCH_SCALED, O.BRANCH_UNSCALED])
def test_algorithm1_update_line(force):
    """mu = 0, wd = 0, no momentum buffer: w <- w - lr * G~ with G~ = gradscale * G (or G)."""
    rng = np.random.default_rng(4)
    numels = [5, 64, 99]
    K = 4
    w = _rand(rng, numels)
    w0 = [a.copy() for a in w]
    g = [_rand(rng, numels, 1e-1) for _ in range(K)]
    mean = [O.replica_mean([g[k][p] for k in range(K)]) for p in range(len(numels))]
    scale = np.array([0.5, 2.0, 1.75], np.float32)
    hp = O.OracleHP(K=K, force_branch=force, has_momentum=False)
    O.ags_step(w, None, g, np.float32(0.1), 0.0, 0.0, hp, scale=scale)
    lr = np.float32(0.1)
    for p in range(len(numels)):
        c = scale[p] if force == O.BRANCH_SCALED else np.float32(1.0)
        assert np.array_equal(w[p], w0[p] - lr * (c * mean[p]))
        assert np.array_equal(g[0][p], mean[p])  # the mean lands in replica 0


def test_update_within_fp32_rounding_of_exact():
    """fp32 result vs the fp64 value of the same formula: within a few ulp of the terms."""
    rng = np.random.default_rng(5)
    n = 4096
    lr, mu, wd = 0.05, 0.9, 5e-4
    w = [rng.standard_normal(n).astype(np.float32)]
    m = [(rng.standard_normal(n) * 1e-2).astype(np.float32)]
    g = [[(rng.standard_normal(n) * 1e-2).astype(np.float32)]]
    scale = np.array([1.5], np.float32)
    w64, m64, g64 = (x[0].astype(np.float64) for x in (w, m, g[0]))
    c = 1.5
    d = c * g64 + np.float64(np.float32(wd)) * w64
    m_new = np.float64(np.float32(mu)) * m64 + d
    w_new = w64 - np.float64(np.float32(lr)) * m_new
    hp = O.OracleHP(K=1, force_branch=O.BRANCH_SCALED)
    O.ags_step(w, m, g, lr, mu, wd, hp, scale=scale)
    mag_m = np.abs(c * g64) + np.abs(wd * w64) + np.abs(mu * m64)
    assert np.all(np.abs(m[0] - m_new) <= 4 * U32 * mag_m)
    assert np.all(np.abs(w[0] - w_new) <= 4 * U32 * (np.abs(w64) + lr * mag_m))
    # every term is visible: each one moves m by far more than the rounding bound
    for term in (np.abs(wd * w64), np.abs(mu * m64), np.abs(c * g64)):
        assert np.median(term / (4 * U32 * mag_m)) > 10


# --------------------------------------------------------------------------
# Hand-worked two-layer example
# --------------------------------------------------------------------------

def _two_layer(g2_prev, steps_done, refresh=False):
    wA = np.array([1.0, 2.0], np.float32)
    wB = np.array([2.0], np.float32)
    gA = [np.array([1.0, 3.0], np.float32), np.array([3.0, 1.0], np.float32)]
    gB = [np.array([0.0], np.float32), np.array([4.0], np.float32)]
    w = [wA, wB]
    m = [np.zeros(2, np.float32), np.zeros(1, np.float32)]
    grads = [[gA[0], gB[0]], [gA[1], gB[1]]]
    scale = np.array([0.5, 2.0], np.float32)
    state = np.array([g2_prev, steps_done, 0, 0], np.float64)
    hp = O.OracleHP(K=2, refresh_scale=refresh)
    stats = O.ags_step(w, m, grads, np.float32(0.1), 0.9, 0.0, hp, scale=scale, state=state)
    return w, m, grads, scale, state, stats


def test_two_layer_example_scaled():
    # mean: gA = [2, 2], gB = [2]; |gA|^2 = 8, |gB|^2 = 4, |G|^2 = 12
    # prev 10: Delta = |12 - 10| / 10 = 0.2 < 0.5 -> scaled with gradscale = [0.5, 2]
    # G~A = [1, 1], G~B = [4]; m = G~ (m was 0); w = w - 0.1 m
    w, m, grads, scale, state, stats = _two_layer(10.0, 5)
    assert np.array_equal(grads[0][0], [2.0, 2.0]) and np.array_equal(grads[0][1], [2.0])
    assert state.tolist() == [12.0, 6.0, pytest.approx(0.2, abs=1e-15), 1.0]
    assert np.array_equal(m[0], [1.0, 1.0]) and np.array_equal(m[1], [4.0])
    assert np.array_equal(w[0], np.float32([1.0, 2.0]) - np.float32(0.1) * np.float32([1.0, 1.0]))
    assert w[0].tolist() == pytest.approx([0.9, 1.9], abs=1e-7)
    assert w[1].tolist() == pytest.approx([1.6], abs=1e-7)
    assert stats[:, 0].tolist() == [5.0, 4.0]       # |w|^2 before the update
    assert stats[:, 1].tolist() == [8.0, 4.0]       # |gbar|^2
    assert stats[:, 2].tolist() == [10.0, 0.0]      # |g_0|^2 (replica 0)
    assert stats[:, 5].tolist() == pytest.approx([math.sqrt(5 / 8), 1.0])
    assert stats[:, 6].tolist() == [0.5, 2.0]       # coefficient applied


def test_two_layer_example_unscaled():
    # prev 4: Delta = |12 - 4| / 4 = 2 >= 0.5 -> unscaled: m = gbar, w = w - 0.1 gbar
    w, m, grads, scale, state, stats = _two_layer(4.0, 5)
    assert state[2] == 2.0 and state[3] == 0.0
    assert np.array_equal(m[0], [2.0, 2.0]) and np.array_equal(m[1], [2.0])
    assert w[0].tolist() == pytest.approx([0.8, 1.8], abs=1e-7)
    assert w[1].tolist() == pytest.approx([1.8], abs=1e-7)
    assert stats[:, 6].tolist() == [1.0, 1.0]


def test_two_layer_example_refresh():
    # UpdateGradScale with g_small = replica 0: |g_0A| = sqrt(10), |gbarA| = sqrt(8);
    # |g_0B| = 0 -> sA = min(sqrt(10) / (sqrt(8) + eps), sqrt(2)) = sqrt(10/8), sB = 0
    w, m, grads, scale, state, stats = _two_layer(10.0, 5, refresh=True)
    assert stats[:, 6].tolist() == [0.5, 2.0]   # this step used the old gradscale
    assert scale[0] == np.float32(math.sqrt(10.0) / (math.sqrt(8.0) + 1e-8))
    assert scale[0] == pytest.approx(1.118034, abs=1e-6)
    assert scale[1] == 0.0
    assert stats[:, 7].tolist() == [float(scale[0]), 0.0]


# --------------------------------------------------------------------------
# UpdateGradScale
# --------------------------------------------------------------------------

def test_scale_elementwise_closed_forms():
    gs = np.array([1.0, -2.0, 0.0, 3.0, 2e-8, 5.0], np.float32)
    gl = np.array([2.0, 1.0, 5.0, -1e-8, 1e-8, -0.5], np.float32)
    s = O.scale_elementwise(gs, gl, 1e-8, 4.0)
    assert s[0] == np.float32(1.0) / (np.float32(2.0) + np.float32(1e-8))
    assert s[1] == 2.0                         # |-2 / 1|
    assert s[2] == 0.0
    assert s[3] == 4.0                         # 3 / (-1e-8 + 1e-8) = inf -> s_max
    assert s[4] == np.float32(1.0)             # eps inside the denominator: 2e-8 / 2e-8
    assert s[5] == 4.0                         # |5 / -0.5| = 10 -> clamped to s_max


def test_scale_tensor_closed_forms():
    assert O.scale_tensor(10.0, 8.0, 1e-8, math.sqrt(2)) == np.float32(
        math.sqrt(10.0) / (math.sqrt(8.0) + 1e-8))
    assert O.scale_tensor(0.0, 0.0, 1e-8, 4.0) == 0.0
    assert O.scale_tensor(4.0, 0.0, 1e-8, 3.0) == 3.0     # 2 / 1e-8 -> clamped
    assert O.scale_tensor(1.0, 4.0, 1e-8, 3.0) == pytest.approx(0.5, rel=1e-7)  # s < 1 allowed
    # eps placement: |g_l| = 1e-8 -> 2e-8 / (1e-8 + 1e-8) = 1, not 2
    assert O.scale_tensor(4e-16, 1e-16, 1e-8, 3.0) == pytest.approx(1.0, rel=1e-6)


def test_scales_bounded_by_smax_lemma1():
    """Lemma 1 needs s_p <= s_max for every parameter: both granularities."""
    rng = np.random.default_rng(6)
    numels = [1, 10, 1000, 3]
    gs = [(rng.standard_normal(n) * 10 ** rng.uniform(-4, 4)).astype(np.float32) for n in numels]
    gl = [(rng.standard_normal(n) * 10 ** rng.uniform(-4, 4)).astype(np.float32) for n in numels]
    for s_max in (1.0, math.sqrt(8), 16.0):
        scale = np.zeros(len(numels), np.float32)
        O.update_scale(gs, gl, 1e-8, s_max, O.GRAN_TENSOR, scale=scale)
        assert np.all(scale <= np.float32(s_max)) and np.all(scale >= 0)
        se = [np.zeros(n, np.float32) for n in numels]
        O.update_scale(gs, gl, 1e-8, s_max, O.GRAN_ELEMENT, scale_elem=se)
        for a in se:
            assert np.all(a <= np.float32(s_max)) and np.all(a >= 0)


def test_iid_replicas_give_sqrt_k_ratio():
    """For i.i.d. replicas E|g_0|^2 / E|gbar|^2 = K: the per-layer refresh lands at ~sqrt(K)."""
    rng = np.random.default_rng(7)
    K, n = 8, 200_000
    g = [[(rng.standard_normal(n) * 1e-3).astype(np.float32)] for _ in range(K)]
    w = [np.zeros(n, np.float32)]
    m = [np.zeros(n, np.float32)]
    scale = np.ones(1, np.float32)
    hp = O.OracleHP(K=K, refresh_scale=True, s_max=100.0)
    stats = O.ags_step(w, m, g, 0.1, 0.9, 0.0, hp, scale=scale)
    assert stats[0, 2] / stats[0, 1] == pytest.approx(K, rel=0.03)
    assert scale[0] == pytest.approx(math.sqrt(K), rel=0.02)


# --------------------------------------------------------------------------
# Rules: static scaling (Eq. 8), LARS (prior art), per-element AGS
# --------------------------------------------------------------------------

def test_static_rule_uses_s_when_scaled():
    rng = np.random.default_rng(8)
    g = [[rng.standard_normal(10).astype(np.float32)]]
    mean = g[0][0].copy()
    w = [np.zeros(10, np.float32)]
    hp = O.OracleHP(K=1, rule=O.RULE_STATIC, static_s=4.0, force_branch=O.BRANCH_SCALED,
                    has_momentum=False)
    stats = O.ags_step(w, None, g, np.float32(1.0), 0.0, 0.0, hp, scale=np.full(1, 9, np.float32))
    assert np.array_equal(w[0], -(np.float32(4.0) * mean))
    assert stats[0, 6] == 4.0


@pytest.mark.parametrize("alpha", [0.5, 2.0, 10.0])
def test_lars_ratio_scales_with_weights(alpha):
    """ratio = |w| / |g|: w -> alpha w multiplies it by alpha; g -> alpha g divides it."""
    rng = np.random.default_rng(9)
    numels = [3, 50, 400]
    w = _rand(rng, numels)
    g = [_rand(rng, numels, 1e-2) for _ in range(2)]
    base = O.layer_stats(w, g)
    w2 = [(a * np.float32(alpha)).astype(np.float32) for a in w]
    scaled_w = O.layer_stats(w2, g)
    g2 = [[(a * np.float32(alpha)).astype(np.float32) for a in r] for r in g]
    scaled_g = O.layer_stats(w, g2)
    assert scaled_w[:, 5] == pytest.approx(alpha * base[:, 5], rel=1e-6)
    assert scaled_g[:, 5] == pytest.approx(base[:, 5] / alpha, rel=1e-6)


def test_lars_rule_coefficient():
    rng = np.random.default_rng(10)
    numels = [20, 30]
    w = _rand(rng, numels)
    w[1][:] = 0.0                                   # zero-norm weights: coefficient falls back to 1
    g = [_rand(rng, numels, 1e-2)]
    sw = [O.sqnorm(a) for a in w]
    sg = [O.sqnorm(a) for a in g[0]]
    hp = O.OracleHP(K=1, rule=O.RULE_LARS, lars_trust=0.02)
    stats = O.ags_step(w, [np.zeros(n, np.float32) for n in numels], g, 0.1, 0.9, 5e-4, hp,
                       scale=np.ones(2, np.float32))
    trust = float(np.float32(0.02))  # the hyper-parameter is fp32
    assert stats[0, 6] == np.float32(trust * (math.sqrt(sw[0]) / math.sqrt(sg[0])))
    assert stats[1, 6] == 1.0


def test_per_element_scaled_step():
    rng = np.random.default_rng(11)
    n = 37
    g = [[rng.standard_normal(n).astype(np.float32)]]
    mean = g[0][0].copy()
    s = [rng.uniform(0, 2, n).astype(np.float32)]
    w = [np.zeros(n, np.float32)]
    hp = O.OracleHP(K=1, granularity=O.GRAN_ELEMENT, force_branch=O.BRANCH_SCALED,
                    has_momentum=False)
    O.ags_step(w, None, g, np.float32(1.0), 0.0, 0.0, hp, scale_elem=s)
    assert np.array_equal(w[0], -(s[0] * mean))


def test_layer_stats_leaves_replicas_untouched():
    rng = np.random.default_rng(12)
    numels = [0, 1, 17]
    w = _rand(rng, numels)
    g = [_rand(rng, numels) for _ in range(3)]
    before = [[a.copy() for a in r] for r in g]
    st = O.layer_stats(w, g)
    for r, rb in zip(g, before):
        for a, b in zip(r, rb):
            assert np.array_equal(a, b)
    assert st[0].tolist() == [0.0] * 8
    mean = O.replica_mean([g[k][2] for k in range(3)])
    assert st[2, 1] == O.sqnorm(mean) and st[2, 0] == O.sqnorm(w[2])


@pytest.mark.parametrize("rule,gran,refresh", [
    (O.RULE_AGS, O.GRAN_TENSOR, True),
    (O.RULE_AGS, O.GRAN_TENSOR, False),
    (O.RULE_LARS, O.GRAN_TENSOR, False),
    (O.RULE_AGS, O.GRAN_ELEMENT, False),
])
def test_threaded_oracle_is_bitwise_the_serial_one(rule, gran, refresh):
    """The CPU baseline on all host cores runs the oracle's per-tensor parts on several threads;
    the norms are still added in tensor order on one thread, so every output (w, m, the mean,
    statistics, state, gradscale) must equal the single-threaded oracle's bit for bit, for any
    thread count, over several steps of both branches."""
    rng = np.random.default_rng(7)
    numels = [int(x) for x in rng.integers(1, 3000, size=37)] + [0, 1, 40000]
    K = 4

    def inputs():
        r = np.random.default_rng(8)
        w = [r.standard_normal(n).astype(np.float32) for n in numels]
        m = [(r.standard_normal(n) * 1e-3).astype(np.float32) for n in numels]
        se = [r.uniform(0.5, 2.0, n).astype(np.float32) for n in numels]
        return w, m, se

    def grads(step, mult):
        r = np.random.default_rng(100 + step)
        return [[(r.standard_normal(n) * 1e-3 * mult).astype(np.float32) for n in numels]
                for _ in range(K)]

    runs = []
    for threads in (None, 1, 2, 5, max(2, O.max_threads())):
        w, m, se = inputs()
        scale = np.linspace(0.5, 1.5, len(numels)).astype(np.float32)
        state = O.new_state()
        hp = O.OracleHP(K=K, rule=rule, granularity=gran, lars_trust=0.01)
        out = []
        for step, mult in ((1, 1.0), (1, 1.0), (2, 2.0)):
            g = grads(step, mult)
            hp.refresh_scale = refresh and step == 1
            stats = O.ags_step(w, m, g, 0.1, 0.9, 5e-4, hp, scale=scale,
                               scale_elem=se if gran == O.GRAN_ELEMENT else None, state=state,
                               threads=threads)
            out.append([np.concatenate(w), np.concatenate(m), np.concatenate(g[0]), stats,
                        state.copy(), scale.copy()])
        runs.append(out)
    assert [int(s[4][3]) for s in runs[0]] == [0, 1, 0]  # both branches
    for other in runs[1:]:
        for a, b in zip(runs[0], other):
            for x, y in zip(a, b):
                assert np.array_equal(x, y, equal_nan=True)
