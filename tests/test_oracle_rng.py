"""Pins for the oracle's random streams and number formats (CPU only).

Philox4x32-10 is pinned word by word by the known-answer vectors published
with Random123 (Salmon et al., SC'11; tests/golden/philox4x32_10_kat.json),
and structurally by inverting it: the inverse below is derived from the
round definition with the Weyl key increments computed here from their
closed forms, 2^32 (golden ratio - 1) and 2^32 (sqrt(3) - 1).
"""
import json
import os
from decimal import Decimal, getcontext

import numpy as np
import pytest
import torch

M32 = 1 << 32
PHILOX_M0, PHILOX_M1 = 0xD2511F53, 0xCD9E8D57   # multipliers published with Philox4x32


def _weyl_constants():
    getcontext().prec = 60
    phi_m1 = (Decimal(5).sqrt() - 1) / 2
    sqrt3_m1 = Decimal(3).sqrt() - 1
    return int(phi_m1 * M32), int(sqrt3_m1 * M32)


def _philox_inverse(out, key):
    """Undo the 10 rounds: lo(M*c) determines c because M is odd."""
    w0, w1 = _weyl_constants()
    inv0, inv1 = pow(PHILOX_M0, -1, M32), pow(PHILOX_M1, -1, M32)
    n0, n1, n2, n3 = (int(v) for v in out)
    for r in reversed(range(10)):
        k0 = (int(key[0]) + r * w0) % M32
        k1 = (int(key[1]) + r * w1) % M32
        c2 = (n1 * inv1) % M32
        hi1 = (PHILOX_M1 * c2) >> 32
        c1 = n0 ^ hi1 ^ k0
        c0 = (n3 * inv0) % M32
        hi0 = (PHILOX_M0 * c0) >> 32
        c3 = n2 ^ hi0 ^ k1
        n0, n1, n2, n3 = c0, c1, c2, c3
    return [n0, n1, n2, n3]


def _kat():
    with open(os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.json")) as f:
        g = json.load(f)
    return [([int(x, 16) for x in v["ctr"]], [int(x, 16) for x in v["key"]], [int(x, 16) for x in v["out"]])
            for v in g["vectors"]]


@pytest.mark.parametrize("k", range(3))
def test_philox_known_answer_vectors(orc, k):
    """The three published philox4x32 10-round vectors, word for word."""
    ctr, key, out = _kat()[k]
    assert [int(w) for w in orc.philox4x32_10(ctr, key)] == out


def test_weyl_constants_closed_form():
    assert _weyl_constants() == (0x9E3779B9, 0xBB67AE85)


@pytest.mark.parametrize("seed", range(6))
def test_philox_inverts_to_counter(orc, seed):
    rng = np.random.default_rng(seed)
    for _ in range(50):
        ctr = rng.integers(0, M32, size=4, dtype=np.uint64).astype(np.uint32)
        key = rng.integers(0, M32, size=2, dtype=np.uint64).astype(np.uint32)
        out = orc.philox4x32_10(ctr, key)
        assert _philox_inverse(out, key) == [int(c) for c in ctr]


def test_philox_uniform_and_distinct(orc):
    words = np.concatenate([orc.philox4x32_10([i, 7, 3, 1], [11, 13]) for i in range(4000)])
    assert len(np.unique(words)) == len(words)
    # chi-square on the top 4 bits: 15 dof, 99.99% quantile ~ 44
    counts = np.bincount(words >> 28, minlength=16)
    exp = len(words) / 16
    assert ((counts - exp) ** 2 / exp).sum() < 44.0
    # neighbouring counters are uncorrelated bitwise (avalanche)
    a = orc.philox4x32_10([0, 0, 0, 0], [0, 0])
    b = orc.philox4x32_10([1, 0, 0, 0], [0, 0])
    flipped = sum(bin(int(x) ^ int(y)).count("1") for x, y in zip(a, b))
    assert 32 < flipped < 96


def test_dropout_counter_layout(orc):
    """keep(row, col) is word col & 3 of Philox at (row, col >> 2, step,
    member << 4 | layer) keyed by the seed, compared against floor(p 2^32)."""
    seed, member, layer, step, p = 0x1234_5678_9ABC_DEF0, 5, 2, 17, 0.3
    T = int(np.floor(np.float64(np.float32(p)) * 2.0 ** 32))
    key = [seed & 0xFFFFFFFF, seed >> 32]
    for row in (0, 1, 255, 1000):
        for col in (0, 1, 2, 3, 4, 127, 130):
            w = orc.philox4x32_10([row, col >> 2, step, (member << 4) | layer], key)[col & 3]
            assert orc.dropout_keep(seed, member, layer, step, row, col, p) == int(w >= T)


def test_dropout_rate_zero_never_drops(orc):
    assert all(orc.dropout_keep(3, 1, 0, s, r, c, 0.0) == 1
               for s in range(3) for r in range(40) for c in range(40))


@pytest.mark.parametrize("p", [0.05, 0.2, 0.5])
def test_dropout_fraction_binomial(orc, p):
    n = 0
    dropped = 0
    for r in range(64):
        for c in range(128):
            dropped += 1 - orc.dropout_keep(99, 3, 1, 4, r, c, p)
            n += 1
    sigma = np.sqrt(n * p * (1 - p))
    assert abs(dropped - n * p) < 5 * sigma


def test_round_bf16_matches_torch(orc):
    rng = np.random.default_rng(0)
    vals = np.concatenate([
        rng.standard_normal(3000).astype(np.float32),
        (rng.standard_normal(500) * 1e-38).astype(np.float32),      # subnormal range
        (rng.standard_normal(500) * 1e30).astype(np.float32),
        np.array([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8, -(1.0 + 2.0 ** -8), 2.0 ** -133,
                  3 * 2.0 ** -134, 0.0, -0.0, 65504.0, 3.3895314e38], dtype=np.float32),
    ])
    ref = torch.from_numpy(vals).to(torch.bfloat16).to(torch.float64).numpy()
    got = np.array([orc.round_bf16(float(v)) for v in vals])
    np.testing.assert_array_equal(got, ref)


def test_init_values(orc):
    seed, member, layer, fan_in = 2, 7, 1, 96
    key = [seed & 0xFFFFFFFF, seed >> 32]
    bound = 1.0 / np.sqrt(fan_in)
    vals = []
    for e in range(2000):
        w = orc.philox4x32_10([e >> 2, 0, 0, (1 << 28) | (member << 4) | layer], key)[e & 3]
        u = ((int(w) >> 8) + 0.5) * 2.0 ** -24
        want = float(np.float32((2 * u - 1) * bound))
        got = orc.init_value(seed, member, layer, e, fan_in)
        assert got == want
        vals.append(got)
    vals = np.array(vals)
    assert np.all(np.abs(vals) <= bound)
    # U(-b, b): mean 0, variance b^2 / 3
    assert abs(vals.mean()) < 5 * bound / np.sqrt(3 * len(vals))
    assert abs(vals.var() / (bound ** 2 / 3) - 1) < 0.1


def test_dropout_mask_equals_elementwise_decisions(orc):
    """The whole-layer mask (one counter per four columns) equals the
    element-by-element decision, including a ragged last column group."""
    seed, member, layer, step, p = 0xDEADBEEF12345678, 9, 3, 41, 0.37
    B, w = 7, 30
    m = orc.dropout_mask(seed, member, layer, step, B, w, p)
    want = np.array([[orc.dropout_keep(seed, member, layer, step, r, c, p) for c in range(w)] for r in range(B)])
    np.testing.assert_array_equal(m, want)
    assert np.all(orc.dropout_mask(seed, member, layer, step, B, w, 0.0) == 1)
