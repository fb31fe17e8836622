"""Seeded synthetic workloads: parameter-set shapes and input fills.

This module is shared by the tests, the benchmark and the smoke check, on both
sides of a parity comparison (CUDA library and CPU oracle).  It holds shapes
and random fills only -- none of the optimizer step's arithmetic.

The paper evaluates on ImageNet/CIFAR/CalTech models (Sec. IV-B); only their
parameter-set shapes matter to the optimizer step, so each workload is the
exact tensor list of a standard architecture, with synthetic values:

* resnet20  CIFAR ResNet-20, 65 tensors, 272,474 params, K = 1
* resnet18  torchvision ResNet-18, 62 tensors, 11,689,512 params, K = 4
* resnet50  torchvision ResNet-50, 161 tensors, 25,557,032 params, K = 8
* vgg16     torchvision VGG-16, 32 tensors, 138,357,544 params, K = 8
* stress    4096 1-D tensors, numel log-uniform in [64, 4Mi] (~1.55e9), K in {1, 4, 16}

Values: conv/fc weights Kaiming-normal (std = sqrt(2 / fan_in)), BatchNorm
gamma = 1 and beta = 0, biases 0 (stress: w ~ N(0, 0.02)); replica gradients
N(0, sigma) times a per-tensor factor f_p (log-uniform, shared by all
replicas); momentum zero or N(0, sigma_m).  Stress tensors with p % 64 == 7
have all-zero gradients, p % 64 == 13 all-zero weights, p % 64 == 21 both.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch

__all__ = ["ParamSet", "param_set", "Workload", "WORKLOADS", "workload", "Buffers",
           "allocate", "fill_state", "fill_grads", "fill_small", "to_numpy", "STEP_MULTIPLIERS"]

# Per-step global multipliers on the gradients of parity runs: steps 1..10.
# A x2 jump multiplies |G|^2 by 4 (Delta ~ 3), a return from it by 1/4
# (Delta ~ 0.75), so both branches of Algorithm 1 occur with Delta far from 0.5.
STEP_MULTIPLIERS = [1.0, 1.0, 1.0, 2.0, 1.0, 1.0, 0.5, 1.0, 1.0, 1.0]

KIND_WEIGHT, KIND_BN_GAMMA, KIND_ZERO, KIND_NORMAL = 0, 1, 2, 3


@dataclass
class ParamSet:
    name: str
    shapes: list = field(default_factory=list)
    kinds: list = field(default_factory=list)

    def add(self, shape, kind):
        self.shapes.append(tuple(int(s) for s in shape))
        self.kinds.append(kind)

    @property
    def numels(self) -> list[int]:
        return [int(np.prod(s)) if len(s) else 1 for s in self.shapes]

    @property
    def n_tensors(self) -> int:
        return len(self.shapes)

    @property
    def n_params(self) -> int:
        return sum(self.numels)


def _conv_bn(ps, cout, cin, k):
    ps.add((cout, cin, k, k), KIND_WEIGHT)
    ps.add((cout,), KIND_BN_GAMMA)
    ps.add((cout,), KIND_ZERO)


def _resnet20() -> ParamSet:
    ps = ParamSet("resnet20")
    _conv_bn(ps, 16, 3, 3)
    cin = 16
    for width in (16, 32, 64):
        for b in range(3):
            _conv_bn(ps, width, cin, 3)
            _conv_bn(ps, width, width, 3)
            if cin != width:
                _conv_bn(ps, width, cin, 1)
            cin = width
    ps.add((10, 64), KIND_WEIGHT)
    ps.add((10,), KIND_ZERO)
    return ps


def _resnet_imagenet(name, block, layers) -> ParamSet:
    ps = ParamSet(name)
    _conv_bn(ps, 64, 3, 7)
    cin = 64
    expansion = 4 if block == "bottleneck" else 1
    for i, (width, n) in enumerate(zip((64, 128, 256, 512), layers)):
        for b in range(n):
            stride_or_grow = b == 0 and (i > 0 or cin != width * expansion)
            if block == "basic":
                _conv_bn(ps, width, cin, 3)
                _conv_bn(ps, width, width, 3)
            else:
                _conv_bn(ps, width, cin, 1)
                _conv_bn(ps, width, width, 3)
                _conv_bn(ps, width * expansion, width, 1)
            if stride_or_grow:
                _conv_bn(ps, width * expansion, cin, 1)
            cin = width * expansion
    ps.add((1000, cin), KIND_WEIGHT)
    ps.add((1000,), KIND_ZERO)
    return ps


def _vgg16() -> ParamSet:
    ps = ParamSet("vgg16")
    cin = 3
    for v in (64, 64, "M", 128, 128, "M", 256, 256, 256, "M", 512, 512, 512, "M",
              512, 512, 512, "M"):
        if v == "M":
            continue
        ps.add((v, cin, 3, 3), KIND_WEIGHT)
        ps.add((v,), KIND_ZERO)
        cin = v
    for fin, fout in ((512 * 7 * 7, 4096), (4096, 4096), (4096, 1000)):
        ps.add((fout, fin), KIND_WEIGHT)
        ps.add((fout,), KIND_ZERO)
    return ps


def _stress(seed=4, n=4096, lo=64, hi=4 * 1024 * 1024) -> ParamSet:
    rng = np.random.default_rng([seed, 1])
    sizes = np.rint(np.exp(rng.uniform(math.log(lo), math.log(hi), size=n))).astype(np.int64)
    ps = ParamSet("stress")
    for s in sizes:
        ps.add((int(s),), KIND_NORMAL)
    return ps


def param_set(name: str, **kw) -> ParamSet:
    if name == "resnet20":
        return _resnet20()
    if name == "resnet18":
        return _resnet_imagenet("resnet18", "basic", (2, 2, 2, 2))
    if name == "resnet50":
        return _resnet_imagenet("resnet50", "bottleneck", (3, 4, 6, 3))
    if name == "vgg16":
        return _vgg16()
    if name == "stress":
        return _stress(**kw)
    raise KeyError(name)


@dataclass
class Workload:
    """One parameter set with its value recipe and optimizer settings."""
    name: str
    K: int
    seed: int
    grad_std: float
    factor_range: tuple | None      # per-tensor log-uniform gradient factor, None = 1
    mom_std: float                   # 0 = zero-initialised momentum
    lr: float = 0.1
    momentum: float = 0.9
    weight_decay: float = 5e-4
    s_max: float | None = None      # None = sqrt(K) (b_small = one replica); K = 1: sqrt(8)
    w_std: float = 0.02             # stress weights
    zero_patterns: bool = False
    small_noise: float = 1e-3       # K = 1: g_small = g + N(0, small_noise)
    stress_n: int = 4096

    @property
    def pset(self) -> ParamSet:
        if self.name.startswith("stress"):
            return _stress(seed=self.seed, n=self.stress_n)
        return param_set(self.name)

    @property
    def smax(self) -> float:
        if self.s_max is not None:
            return self.s_max
        return math.sqrt(self.K) if self.K > 1 else math.sqrt(8.0)


WORKLOADS = {
    "resnet20": Workload("resnet20", K=1, seed=0, grad_std=1e-3, factor_range=(0.1, 10.0), mom_std=0.0),
    "resnet18": Workload("resnet18", K=4, seed=1, grad_std=1e-3, factor_range=None, mom_std=0.0),
    "resnet50": Workload("resnet50", K=8, seed=2, grad_std=1e-3, factor_range=(0.01, 100.0), mom_std=1e-3),
    "vgg16": Workload("vgg16", K=8, seed=3, grad_std=1e-4, factor_range=None, mom_std=0.0),
    "stress_k1": Workload("stress", K=1, seed=4, grad_std=1.0, factor_range=(1e-6, 1e2), mom_std=0.0,
                          zero_patterns=True),
    "stress_k4": Workload("stress", K=4, seed=4, grad_std=1.0, factor_range=(1e-6, 1e2), mom_std=0.0,
                          zero_patterns=True),
    "stress_k16": Workload("stress", K=16, seed=4, grad_std=1.0, factor_range=(1e-6, 1e2), mom_std=0.0,
                           zero_patterns=True),
}


def workload(name: str, **overrides) -> Workload:
    w = WORKLOADS[name]
    if overrides:
        w = Workload(**{**w.__dict__, **overrides})
    return w


def _factors(wl: Workload, pset: ParamSet) -> np.ndarray:
    rng = np.random.default_rng([wl.seed, 2])
    n = pset.n_tensors
    if wl.factor_range is None:
        f = np.ones(n)
    else:
        lo, hi = wl.factor_range
        f = np.exp(rng.uniform(math.log(lo), math.log(hi), size=n))
    if wl.zero_patterns:
        p = np.arange(n)
        f[(p % 64 == 7) | (p % 64 == 21)] = 0.0
    return f


@dataclass
class Buffers:
    """Device (or host) tensors of one workload, each role in one flat buffer.

    Tensor p of every role starts at element offsets[p] of its flat buffer;
    offsets are multiples of ``align`` elements (default 64 = 256 bytes, the
    alignment separate allocations would have), plus ``shift`` elements to
    build deliberately misaligned views."""
    pset: ParamSet
    offsets: list
    total: int
    w_flat: torch.Tensor
    m_flat: torch.Tensor | None
    g_flats: list
    w: list
    m: list | None
    g: list                 # g[k][p]
    factors: np.ndarray     # per-tensor gradient factor f_p

    @property
    def numels(self):
        return self.pset.numels


def _layout(numels, align, shift):
    offs, o = [], shift
    for n in numels:
        offs.append(o)
        o += n
        if align > 1:
            o = (o + align - 1) // align * align
    return offs, o


def _views(flat, offsets, shapes, numels):
    return [flat[o:o + n].view(s) if len(s) else flat[o:o + n].view(()) for o, n, s in
            zip(offsets, numels, shapes)]


def allocate(wl: Workload, device="cpu", K: int | None = None, align: int = 64, shift: int = 0,
             with_momentum: bool = True, pset: ParamSet | None = None) -> Buffers:
    pset = pset or wl.pset
    K = wl.K if K is None else K
    numels = pset.numels
    offsets, total = _layout(numels, align, shift)
    mk = lambda: torch.zeros(max(total, 1), dtype=torch.float32, device=device)  # noqa: E731
    w_flat = mk()
    m_flat = mk() if with_momentum else None
    g_flats = [mk() for _ in range(K)]
    return Buffers(pset, offsets, total, w_flat, m_flat, g_flats,
                   _views(w_flat, offsets, pset.shapes, numels),
                   _views(m_flat, offsets, pset.shapes, numels) if with_momentum else None,
                   [_views(f, offsets, pset.shapes, numels) for f in g_flats],
                   _factors(wl, pset))


def _gen(device, *key):
    g = torch.Generator(device=device)
    h = 0
    for k in key:
        h = (h * 1_000_003 + int(k) + 1) % (2 ** 62)
    g.manual_seed(h)
    return g


def _per_tensor(buf: Buffers, values, device) -> torch.Tensor:
    """Expand one value per tensor to the flat layout (padding gets 0)."""
    counts, vals, pos = [], [], 0
    for o, n, v in zip(buf.offsets, buf.numels, values):
        if o > pos:
            counts.append(o - pos)
            vals.append(0.0)
        counts.append(n)
        vals.append(float(v))
        pos = o + n
    size = max(buf.total, 1)
    if size > pos:
        counts.append(size - pos)
        vals.append(0.0)
    return torch.repeat_interleave(torch.tensor(vals, dtype=torch.float32, device=device),
                                   torch.tensor(counts, dtype=torch.int64, device=device),
                                   output_size=size)


def fill_state(buf: Buffers, wl: Workload) -> None:
    """w: Kaiming-normal / BN gamma 1 / zeros (stress: N(0, w_std)); m: 0 or N(0, mom_std)."""
    device = buf.w_flat.device
    pset = buf.pset
    std = np.zeros(pset.n_tensors)
    const = np.zeros(pset.n_tensors)
    for p, (shape, kind) in enumerate(zip(pset.shapes, pset.kinds)):
        if kind == KIND_WEIGHT:
            fan_in = int(np.prod(shape[1:]))
            std[p] = math.sqrt(2.0 / fan_in)
        elif kind == KIND_BN_GAMMA:
            const[p] = 1.0
        elif kind == KIND_NORMAL:
            std[p] = wl.w_std
            if wl.zero_patterns and (p % 64 == 13 or p % 64 == 21):
                std[p] = 0.0
    torch.randn(buf.w_flat.shape, generator=_gen(device, wl.seed, 1), device=device, out=buf.w_flat)
    buf.w_flat.mul_(_per_tensor(buf, std, device)).add_(_per_tensor(buf, const, device))
    if buf.m_flat is not None:
        if wl.mom_std > 0:
            torch.randn(buf.m_flat.shape, generator=_gen(device, wl.seed, 2), device=device,
                        out=buf.m_flat)
            buf.m_flat.mul_(_per_tensor(buf, np.full(pset.n_tensors, wl.mom_std), device))
        else:
            buf.m_flat.zero_()


def fill_grads(buf: Buffers, wl: Workload, step: int = 0, multiplier: float = 1.0) -> None:
    """Replica gradients of one step: N(0, grad_std) * f_p * multiplier, fresh per (seed, step, k)."""
    device = buf.w_flat.device
    fac = _per_tensor(buf, buf.factors * wl.grad_std * multiplier, device)
    for k, flat in enumerate(buf.g_flats):
        torch.randn(flat.shape, generator=_gen(device, wl.seed, 3, step, k), device=device, out=flat)
        flat.mul_(fac)


def fill_small(buf: Buffers, wl: Workload, out_flat: torch.Tensor, step: int = 0) -> None:
    """A small-batch gradient for K = 1: replica 0 plus N(0, small_noise) on non-zero tensors."""
    device = out_flat.device
    torch.randn(out_flat.shape, generator=_gen(device, wl.seed, 4, step), device=device, out=out_flat)
    mask = _per_tensor(buf, (buf.factors != 0).astype(np.float64) * wl.small_noise, device)
    out_flat.mul_(mask).add_(buf.g_flats[0])


def to_numpy(tensors) -> list:
    """Host float32 copies (contiguous, writeable) of a list of tensors."""
    return [t.detach().reshape(-1).cpu().numpy().copy() for t in tensors]
