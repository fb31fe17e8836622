"""The exchange of a sharded step on CPU: two gloo ranks, no GPU.

In a step sharded over ranks (tula_ags_shard_reduce / tula_ags_shard_update) the only data the
ranks exchange is their share of |G|^2 (Eq. 5): TULA_G2_SHARE_WORDS 64-bit integers -- 32-bit
digits from 2^-352 with carries in the high halves, then a count of inf partials and one of NaN
partials.  combine_g2_shares adds the shares over the process group with an integer SUM.  These
tests encode shares from known partial sums (the documented format, written out here), combine
them with gloo ranks, and check that the combined share decodes to the exact sum of every
rank's partials rounded once to fp64, in any order of addition, with inf and NaN carried.
"""
import math
import os
import socket
from fractions import Fraction

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from paper_2603_18112_gb300 import tula_ags as T

WORDS, DIGITS, BASE = T.TULA_G2_SHARE_WORDS, 21, -352


def encode(values):
    """A share holding the exact sum of non-negative floats (inf and NaN counted)."""
    words = [0] * WORDS
    for v in values:
        if math.isnan(v):
            words[DIGITS + 1] += 1
            continue
        if math.isinf(v):
            words[DIGITS] += 1
            continue
        if v == 0.0:
            continue
        m, e = math.frexp(v)                 # v = m * 2^e, 0.5 <= m < 1
        mi, E = int(m * 2 ** 53), e - 53     # exact: v = mi * 2^E
        s = E - BASE
        assert s >= 0
        x = mi << (s % 32)
        i = s // 32
        while x:
            words[i] += x & 0xffffffff
            x >>= 32
            i += 1
    return torch.tensor([w - (1 << 64) if w >= (1 << 63) else w for w in words], dtype=torch.int64)


def decode(share):
    """The value of a share, rounded once to fp64 (Fraction -> float rounds to nearest even)."""
    w = [int(x) % (1 << 64) for x in share.tolist()]
    if w[DIGITS + 1]:
        return math.nan
    if w[DIGITS]:
        return math.inf
    total = sum(Fraction(w[i]) * Fraction(2) ** (32 * i + BASE) for i in range(DIGITS))
    return float(total)


def exact(values):
    return float(sum(Fraction(v) for v in values))


def _partials(rank, seed, special=None):
    rng = np.random.default_rng([seed, rank])
    # fp32 tile sums over a wide range of magnitudes, and fp64 ones
    v = [float(np.float32(x)) for x in np.exp(rng.uniform(-60, 60, size=300))]
    v += [float(x) for x in np.exp(rng.uniform(-200, 180, size=50))]
    if special and rank == 1:
        v.append(special)
    return v


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, seed, special, out_path):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        share = encode(_partials(rank, seed, special))
        T.combine_g2_shares(share)
        everything = [x for r in range(world) for x in _partials(r, seed, special)]
        got, want = decode(share), (exact(everything) if special is None else special)
        with open(f"{out_path}.{rank}", "w") as f:
            f.write(repr((got, want, share.tolist())))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("special", [None, math.inf, math.nan])
def test_two_ranks_combine_to_the_exact_total(tmp_path, special):
    world = 2
    out = str(tmp_path / "res")
    mp.spawn(_rank_main, args=(world, _free_port(), 5, special, out), nprocs=world, join=True)
    results = [eval(open(f"{out}.{r}").read(), {"inf": math.inf, "nan": math.nan}) for r in range(world)]
    for got, want, _ in results:
        if special is not None and math.isnan(special):
            assert math.isnan(got)
        else:
            assert got == want
    assert results[0][2] == results[1][2]  # every rank holds the same total, word for word


def test_shares_add_in_any_order_and_wrap_harmlessly():
    parts = [_partials(r, 9) for r in range(5)]
    shares = [encode(p) for p in parts]
    total = exact([x for p in parts for x in p])
    for order in ([0, 1, 2, 3, 4], [4, 2, 0, 3, 1], [3, 1, 4, 0, 2]):
        s = torch.zeros(WORDS, dtype=torch.int64)
        for i in order:
            s += shares[i]
        assert decode(s) == total
        assert torch.equal(s, encode([x for p in parts for x in p]))
    # a word past 2^63 is negative in int64; sums still wrap to the right 64-bit pattern
    big = torch.zeros(WORDS, dtype=torch.int64)
    big[3] = (1 << 63) - 5
    s = big + big
    assert int(s[3]) % (1 << 64) == 2 * ((1 << 63) - 5)
