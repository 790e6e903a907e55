"""Pins of the oracle's periodic feature embeddings (App. "Feature
Embeddings": feature j becomes alpha_j * [x_j, cos(w_j x_j + b_j)] + beta_j
and layer 1 reads the d_in embeddings side by side).

* Wiring: with alpha selecting one component per feature, the pack equals a
  plain pack (no embeddings) fed that component as its input and holding the
  matching columns of W_1 -- the x component (d_emb = 1 and 3) and a cosine
  component -- so the column layout j * d_emb + k and the component order are
  fixed.
* Gradients: central finite differences (fp64, p = 0) of the mean loss on
  every embedding parameter (w, b, alpha, beta) of a member with d_emb = 3.
"""
import numpy as np
import pytest

import oracle
from workloads import random_pack


def data(n, d_in, d_out, seed):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((n, d_in)).astype(np.float32)
    y = rng.integers(0, d_out, n).astype(np.int32)
    return X, y


def emb_pack(hp, d_in, d_out, d_emb, freq, seed=2):
    return oracle.OraclePack(d_in, d_out, "multiclass", hp["depth"], hp["width"], hp["dropout"], hp["lr"],
                             hp["wd"], seed=seed, d_emb=d_emb, freq=freq)


def plain_pack(hp, d_in, d_out, seed=2):
    return oracle.OraclePack(d_in, d_out, "multiclass", hp["depth"], hp["width"], hp["dropout"], hp["lr"],
                             hp["wd"], seed=seed)


def copy_params(src, dst, member, L, W0=None):
    for l in range(L + 1):
        W, b = src.get_params(member, l)
        dst.set_params(member, l, W if (l or W0 is None) else W0, b)


@pytest.mark.parametrize("d", [1, 3])
def test_x_component_reproduces_the_plain_pack(d):
    d_in, d_out = 4, 3
    hp = random_pack(1, d_in, d_out, seed=5, dropout=(0.0, 0.0))
    rng = np.random.default_rng(1)
    e = emb_pack(hp, d_in, d_out, [d], rng.standard_normal(d_in * (d - 1)))
    alpha = np.zeros((d_in, d)); alpha[:, 0] = 1.0
    e.set_emb(0, rng.standard_normal((d_in, d - 1)), rng.standard_normal((d_in, d - 1)), alpha, np.zeros((d_in, d)))
    p = plain_pack(hp, d_in, d_out)
    L = int(hp["depth"][0])
    W0 = e.get_params(0, 0)[0][:, 0::d]          # the x columns
    copy_params(e, p, 0, L, W0=W0)
    X, y = data(30, d_in, d_out, 2)
    idx = np.arange(12, dtype=np.int32)
    np.testing.assert_allclose(e.train_step(X, idx, y, 0, update=False), p.train_step(X, idx, y, 0, update=False),
                               rtol=0, atol=1e-14)
    np.testing.assert_allclose(e.get_grads(0, 0)[0][:, 0::d], p.get_grads(0, 0)[0], rtol=0, atol=1e-14)
    if d == 1:   # d_emb = 1 with alpha = 1: the same initial W_1 (same fan-in and counters)
        np.testing.assert_array_equal(e.get_params(0, 0)[0], plain_pack(hp, d_in, d_out).get_params(0, 0)[0])


def test_cosine_component_wiring():
    d_in, d_out, d = 4, 2, 3
    hp = random_pack(1, d_in, d_out, seed=8, dropout=(0.0, 0.0))
    rng = np.random.default_rng(3)
    w = rng.standard_normal((d_in, d - 1))
    b = rng.standard_normal((d_in, d - 1))
    alpha = np.zeros((d_in, d)); alpha[:, 2] = 0.7
    beta = np.zeros((d_in, d)); beta[:, 2] = -0.2
    e = emb_pack(hp, d_in, d_out, [d], w.ravel())
    e.set_emb(0, w, b, alpha, beta)
    X, y = data(25, d_in, d_out, 4)
    # the plain pack sees feature j as 0.7 cos(w_j1 x_j + b_j1) - 0.2
    Xc = (0.7 * np.cos(w[:, 1][None, :] * X.astype(np.float64) + b[:, 1][None, :]) - 0.2).astype(np.float32)
    p = plain_pack(hp, d_in, d_out)
    L = int(hp["depth"][0])
    copy_params(e, p, 0, L, W0=e.get_params(0, 0)[0][:, 2::d])
    idx = np.arange(10, dtype=np.int32)
    le = e.train_step(X, idx, y, 0, update=False)
    lp = p.train_step(Xc, idx, y, 0, update=False)
    assert abs(le[0] - lp[0]) < 1e-6   # Xc went through fp32


def test_embedding_gradients_by_finite_differences():
    d_in, d_out, d = 3, 3, 3
    hp = random_pack(1, d_in, d_out, seed=11, dropout=(0.0, 0.0), width=(16, 32, 16))
    rng = np.random.default_rng(6)
    e = emb_pack(hp, d_in, d_out, [d], rng.standard_normal(d_in * (d - 1)))
    parts = [rng.standard_normal((d_in, d - 1)), rng.standard_normal((d_in, d - 1)),
             rng.standard_normal((d_in, d)), rng.standard_normal((d_in, d)) * 0.3]
    e.set_emb(0, *parts)
    X, y = data(20, d_in, d_out, 7)
    idx = np.arange(20, dtype=np.int32)
    e.train_step(X, idx, y, 0, update=False)
    grads = e.emb(0, grads=True)
    h = 1e-6
    for pi in range(4):
        for pos in np.ndindex(parts[pi].shape):
            vals = []
            for sgn in (+1, -1):
                q = [a.copy() for a in parts]
                q[pi][pos] += sgn * h
                e.set_emb(0, *q)
                vals.append(e.train_step(X, idx, y, 0, update=False)[0])
            fd = (vals[0] - vals[1]) / (2 * h)
            assert abs(fd - grads[pi][pos]) <= 1e-6 * max(1.0, abs(fd)), (pi, pos, fd, grads[pi][pos])
    e.set_emb(0, *parts)


def test_embeddings_train_with_adamw():
    """One update moves alpha (its gradient is non-zero from the zero start)
    and keeps b and w in place while alpha is still zero."""
    d_in, d_out, d = 3, 2, 4
    hp = random_pack(2, d_in, d_out, seed=12, dropout=(0.0, 0.0))
    rng = np.random.default_rng(2)
    freq = rng.standard_normal(2 * d_in * (d - 1))
    e = emb_pack(hp, d_in, d_out, [d, d], freq)
    w0, b0, a0, be0 = e.emb(1)
    np.testing.assert_array_equal(w0.ravel(), freq[d_in * (d - 1):])
    assert not a0.any() and not b0.any() and not be0.any()
    X, y = data(30, d_in, d_out, 9)
    e.train_step(X, np.arange(30, dtype=np.int32), y, 0)
    w1, b1, a1, be1 = e.emb(1)
    assert np.abs(a1).max() > 0 and np.abs(be1).max() > 0
    # zero gradient while alpha is zero: only the decoupled weight decay acts on w
    np.testing.assert_allclose(w1, w0 - float(hp["lr"][1]) * float(hp["wd"][1]) * w0, rtol=1e-15, atol=0)
    assert not b1.any()


def test_embedding_weight_decay_follows_the_bias_flag():
    """The embedding parameters take weight decay as the biases do: with
    wd_on_bias off, a step from alpha = 0 (zero gradient for w and b) leaves
    w exactly in place; with it on, w shrinks by lr wd w."""
    d_in, d_out, d = 3, 2, 4
    hp = random_pack(1, d_in, d_out, seed=13, dropout=(0.0, 0.0))
    freq = np.random.default_rng(4).standard_normal(d_in * (d - 1))
    X, y = data(30, d_in, d_out, 10)
    for on in (False, True):
        e = oracle.OraclePack(d_in, d_out, "multiclass", hp["depth"], hp["width"], hp["dropout"], hp["lr"],
                              hp["wd"], seed=2, wd_on_bias=on, d_emb=[d], freq=freq)
        w0 = e.emb(0)[0].copy()
        e.train_step(X, np.arange(30, dtype=np.int32), y, 0)
        w1 = e.emb(0)[0]
        expect = w0 - float(hp["lr"][0]) * float(hp["wd"][0]) * w0 if on else w0
        np.testing.assert_allclose(w1, expect, rtol=1e-15, atol=0)


@pytest.mark.parametrize("bf16", [False, True])
def test_packed_embedding_members_equal_solo_members(bf16):
    """Members with periodic embeddings of different sizes are independent
    (Sec. 3.6): three AdamW steps of the pack give each member exactly what
    training it alone gives (losses, every parameter, embeddings included,
    and predictions), with the frequencies split member by member."""
    m, d_in, d_out = 4, 5, 3
    hp = random_pack(m, d_in, d_out, seed=19)
    d_emb = np.array([1, 3, 8, 5], dtype=np.int32)
    freq = np.random.default_rng(7).standard_normal(d_in * int(np.sum(d_emb - 1)))
    starts = np.concatenate([[0], np.cumsum(d_in * (d_emb - 1))])
    X, y = data(64, d_in, d_out, 3)
    kw = dict(seed=8, bf16_storage=bf16)
    packed = oracle.OraclePack(d_in, d_out, "multiclass", hp["depth"], hp["width"], hp["dropout"], hp["lr"],
                               hp["wd"], d_emb=d_emb, freq=freq, **kw)
    solos = [oracle.OraclePack(d_in, d_out, "multiclass", hp["depth"][i:i + 1], hp["width"][i:i + 1],
                               hp["dropout"][i:i + 1], hp["lr"][i:i + 1], hp["wd"][i:i + 1], member_id=[i],
                               d_emb=d_emb[i:i + 1], freq=freq[starts[i]:starts[i + 1]], **kw) for i in range(m)]
    rng = np.random.default_rng(1)
    for step in range(3):
        idx = rng.choice(64, 24, replace=False).astype(np.int32)
        lp = packed.train_step(X, idx, y, step)
        for i in range(m):
            assert lp[i] == solos[i].train_step(X, idx, y, step)[0]
    for i in range(m):
        for l in range(int(hp["depth"][i]) + 1):
            for a, b in zip(packed.get_params(i, l), solos[i].get_params(0, l)):
                np.testing.assert_array_equal(a, b)
        for a, b in zip(packed.emb(i), solos[i].emb(0)):
            np.testing.assert_array_equal(a, b)
    Pp = packed.predict(X[:10])
    for i in range(m):
        np.testing.assert_array_equal(Pp[i], solos[i].predict(X[:10])[0])
