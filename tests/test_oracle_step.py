"""Pins for the oracle's training step, validation predictions and AdamW.

The oracle is checked against things other than itself:
  * torch CPU fp64 ``nn.functional.linear`` / ``relu`` + autograd + the
    library losses (cross-entropy, BCE-with-logits, MSE) + ``torch.optim.AdamW``
    (library routines), fed the oracle's dropout masks;
  * central finite differences of the oracle's own loss (pins the backward
    against the forward);
  * the packed pack versus each member trained alone (Sec. 3.6: members are
    trained independently, only their losses are summed);
  * closed forms of the losses at zero weights.
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from workloads import random_pack



class _RoundBF16(torch.autograd.Function):
    """Forward: round to bf16; backward: identity (a stored copy)."""

    @staticmethod
    def forward(ctx, x):
        return x.to(torch.float32).to(torch.bfloat16).to(torch.float64)

    @staticmethod
    def backward(ctx, g):
        return g


class _RoundGradBF16(torch.autograd.Function):
    """Forward: identity; backward: the incoming gradient is stored in bf16."""

    @staticmethod
    def forward(ctx, x):
        return x.clone()

    @staticmethod
    def backward(ctx, g):
        return g.to(torch.float32).to(torch.bfloat16).to(torch.float64)


def _make_data(task, n, d_in, d_out, seed):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((n, d_in)).astype(np.float32)
    if task == "regression":
        y = rng.standard_normal(n).astype(np.float32)
    elif task == "binary":
        y = rng.integers(0, 2, n).astype(np.int32)
    else:
        y = rng.integers(0, d_out, n).astype(np.int32)
    return X, y


class TorchMember:
    """One base MLP in plain torch fp64, initialised from the oracle."""

    def __init__(self, pack, i, lr, wd, p, bf16):
        self.L = int(pack.depth[i])
        self.p = float(np.float32(p))
        self.bf16 = bf16
        self.params = []
        for l in range(self.L + 1):
            W, b = pack.get_params(i, l)
            self.params.append((torch.tensor(W, requires_grad=True), torch.tensor(b, requires_grad=True)))
        flat = [t for pair in self.params for t in pair]
        self.opt = torch.optim.AdamW(flat, lr=float(np.float32(lr)), betas=(0.9, 0.999), eps=1e-8,
                                     weight_decay=float(np.float32(wd)))

    def forward(self, x, masks):
        r = _RoundBF16.apply if self.bf16 else (lambda t: t)
        rg = _RoundGradBF16.apply if self.bf16 else (lambda t: t)
        h = r(x)
        for l in range(self.L):
            W, b = self.params[l]
            z = rg(F.linear(h, r(W), b))
            h = r(F.relu(z) * masks[l] / (1.0 - self.p))
        W, b = self.params[self.L]
        return F.linear(h, W, b)

    def step(self, x, yb, task, masks):
        self.opt.zero_grad()
        logits = self.forward(x, masks)
        if task == "multiclass":
            loss = F.cross_entropy(logits, yb.long())
        elif task == "binary":
            loss = F.binary_cross_entropy_with_logits(logits[:, 0], yb.double())
        else:
            loss = F.mse_loss(logits[:, 0], yb.double())
        loss.backward()
        grads = [(W.grad.clone(), b.grad.clone()) for W, b in self.params]
        self.opt.step()
        return loss.item(), logits.detach(), grads


def _rel(a, b):
    a, b = np.asarray(a, dtype=np.float64), np.asarray(b, dtype=np.float64)
    scale = max(np.abs(b).max(), 1e-300)
    return np.abs(a - b).max() / scale


@pytest.mark.parametrize("task,d_out", [("binary", 1), ("multiclass", 5), ("regression", 1)])
@pytest.mark.parametrize("same_hp", [False, True])
@pytest.mark.parametrize("bf16", [False, True])
def test_oracle_matches_torch_autograd_adamw(orc, task, d_out, same_hp, bf16):
    m, d_in, B, steps = 4, 12, 24, 4
    hp = random_pack(m, d_in, d_out, seed=11 + d_out)
    if same_hp:   # identical hyperparameters: a plain MLP ensemble
        for k in hp:
            hp[k][:] = hp[k][0]
    pack = orc.OraclePack(d_in, d_out, task, hp["depth"], hp["width"], hp["dropout"], hp["lr"],
                          hp["wd"], seed=5, bf16_storage=bf16)
    ref = [TorchMember(pack, i, hp["lr"][i], hp["wd"][i], hp["dropout"][i], bf16) for i in range(m)]
    X, y = _make_data(task, 80, d_in, d_out, seed=3)
    rng = np.random.default_rng(4)
    tol = 1e-9 if not bf16 else 1e-6
    for step in range(steps):
        idx = rng.choice(80, B, replace=False).astype(np.int32)
        losses = pack.train_step(X, idx, y, step)
        for i in range(m):
            masks = [torch.tensor(pack.keep(i, l), dtype=torch.float64) for l in range(int(hp["depth"][i]))]
            loss_t, logits_t, grads_t = ref[i].step(torch.tensor(X[idx], dtype=torch.float64),
                                                    torch.tensor(y[idx]), task, masks)
            assert abs(losses[i] - loss_t) <= tol * max(1.0, abs(loss_t))
            assert _rel(pack.logits(i), logits_t.numpy()) < tol
            for l in range(int(hp["depth"][i]) + 1):
                gW, gb = pack.get_grads(i, l)
                assert _rel(gW, grads_t[l][0].numpy()) < tol, (i, l)
                assert _rel(gb, grads_t[l][1].numpy()) < tol, (i, l)
                W, b = pack.get_params(i, l)
                assert _rel(W, ref[i].params[l][0].detach().numpy()) < tol, (i, l)
                assert _rel(b, ref[i].params[l][1].detach().numpy()) < tol, (i, l)


def test_oracle_adam_state_matches_torch(orc):
    m, d_in = 2, 6
    hp = random_pack(m, d_in, 1, seed=2)
    pack = orc.OraclePack(d_in, 1, "regression", hp["depth"], hp["width"], hp["dropout"], hp["lr"],
                          hp["wd"], seed=9)
    ref = TorchMember(pack, 0, hp["lr"][0], hp["wd"][0], hp["dropout"][0], False)
    X, y = _make_data("regression", 32, d_in, 1, seed=1)
    idx = np.arange(32, dtype=np.int32)
    for step in range(3):
        pack.train_step(X, idx, y, step)
        masks = [torch.tensor(pack.keep(0, l), dtype=torch.float64) for l in range(int(hp["depth"][0]))]
        ref.step(torch.tensor(X, dtype=torch.float64), torch.tensor(y), "regression", masks)
    for l in range(int(hp["depth"][0]) + 1):
        mW, vW, mb, vb = pack.get_adam_state(0, l)
        st = ref.opt.state[ref.params[l][0]]
        assert _rel(mW, st["exp_avg"].numpy()) < 1e-12
        assert _rel(vW, st["exp_avg_sq"].numpy()) < 1e-12
    assert pack.member_steps(0) == 3


@pytest.mark.parametrize("task,d_out", [("binary", 1), ("multiclass", 3), ("regression", 1)])
@pytest.mark.parametrize("p", [0.0, 0.35])
def test_oracle_finite_differences(orc, task, d_out, p):
    d_in, B = 5, 10
    depth, width = [2], [8]
    pack = orc.OraclePack(d_in, d_out, task, depth, width, [p], [1e-3], [1e-3], seed=21)
    X, y = _make_data(task, B, d_in, d_out, seed=7)
    idx = np.arange(B, dtype=np.int32)
    step = 3  # the mask is a fixed function of the step, so it stays fixed under perturbation
    pack.train_step(X, idx, y, step, update=False)
    h = 1e-6
    for l in range(3):
        gW, gb = pack.get_grads(0, l)
        W0, b0 = pack.get_params(0, l)
        rng = np.random.default_rng(l)
        for _ in range(6):
            r, c = rng.integers(0, W0.shape[0]), rng.integers(0, W0.shape[1])
            vals = []
            for s in (+1, -1):
                W = W0.copy()
                W[r, c] += s * h
                pack.set_params(0, l, W, b0)
                vals.append(pack.train_step(X, idx, y, step, update=False)[0])
            pack.set_params(0, l, W0, b0)
            fd = (vals[0] - vals[1]) / (2 * h)
            assert abs(fd - gW[r, c]) <= 1e-6 * max(1.0, abs(fd)), (l, r, c, fd, gW[r, c])
        r = rng.integers(0, b0.shape[0])
        vals = []
        for s in (+1, -1):
            b = b0.copy()
            b[r] += s * h
            pack.set_params(0, l, W0, b)
            vals.append(pack.train_step(X, idx, y, step, update=False)[0])
        pack.set_params(0, l, W0, b0)
        assert abs((vals[0] - vals[1]) / (2 * h) - gb[r]) <= 1e-6


@pytest.mark.parametrize("bf16", [False, True])
def test_packed_equals_solo_members(orc, bf16):
    m, d_in, d_out = 5, 9, 4
    hp = random_pack(m, d_in, d_out, seed=17)
    X, y = _make_data("multiclass", 64, d_in, d_out, seed=2)
    packed = orc.OraclePack(d_in, d_out, "multiclass", hp["depth"], hp["width"], hp["dropout"],
                            hp["lr"], hp["wd"], seed=8, bf16_storage=bf16)
    solos = [orc.OraclePack(d_in, d_out, "multiclass", hp["depth"][i:i + 1], hp["width"][i:i + 1],
                            hp["dropout"][i:i + 1], hp["lr"][i:i + 1], hp["wd"][i:i + 1], seed=8,
                            bf16_storage=bf16, member_id=[i]) for i in range(m)]
    rng = np.random.default_rng(0)
    for step in range(3):
        idx = rng.choice(64, 20, replace=False).astype(np.int32)
        lp = packed.train_step(X, idx, y, step)
        for i in range(m):
            ls = solos[i].train_step(X, idx, y, step)
            assert lp[i] == ls[0]
    for i in range(m):
        for l in range(int(hp["depth"][i]) + 1):
            Wp, bp = packed.get_params(i, l)
            Ws, bs = solos[i].get_params(0, l)
            np.testing.assert_array_equal(Wp, Ws)
            np.testing.assert_array_equal(bp, bs)
    Pp = packed.predict(X[:10])
    for i in range(m):
        np.testing.assert_array_equal(Pp[i], solos[i].predict(X[:10])[0])


@pytest.mark.parametrize("bf16", [False, True])
def test_stacked_batches_equal_solo_members_on_their_own_batches(orc, bf16):
    """Sec. 3.6: each base model trains on its own batch sequence; a stacked
    step (idx [m, B]) gives member i exactly what training it alone on row i
    of idx gives (and a shifted or transposed row would not)."""
    m, d_in, d_out = 4, 7, 3
    hp = random_pack(m, d_in, d_out, seed=23)
    X, y = _make_data("multiclass", 80, d_in, d_out, seed=5)
    packed = orc.OraclePack(d_in, d_out, "multiclass", hp["depth"], hp["width"], hp["dropout"],
                            hp["lr"], hp["wd"], seed=9, bf16_storage=bf16)
    solos = [orc.OraclePack(d_in, d_out, "multiclass", hp["depth"][i:i + 1], hp["width"][i:i + 1],
                            hp["dropout"][i:i + 1], hp["lr"][i:i + 1], hp["wd"][i:i + 1], seed=9,
                            bf16_storage=bf16, member_id=[i]) for i in range(m)]
    rng = np.random.default_rng(1)
    for step in range(3):
        idx = np.stack([rng.choice(80, 16, replace=False) for _ in range(m)]).astype(np.int32)
        lp = packed.train_step(X, idx, y, step)
        for i in range(m):
            assert lp[i] == solos[i].train_step(X, idx[i], y, step)[0]
    for i in range(m):
        for l in range(int(hp["depth"][i]) + 1):
            np.testing.assert_array_equal(packed.get_params(i, l)[0], solos[i].get_params(0, l)[0])
            np.testing.assert_array_equal(packed.get_params(i, l)[1], solos[i].get_params(0, l)[1])


def test_stacked_batches_with_one_batch_equal_the_shared_step(orc):
    m, d_in, d_out = 3, 6, 1
    hp = random_pack(m, d_in, d_out, seed=31)
    X, y = _make_data("regression", 50, d_in, d_out, seed=6)
    a = orc.OraclePack(d_in, d_out, "regression", hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"], seed=4)
    b = orc.OraclePack(d_in, d_out, "regression", hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"], seed=4)
    rng = np.random.default_rng(2)
    for step in range(2):
        idx = rng.choice(50, 12, replace=False).astype(np.int32)
        np.testing.assert_array_equal(a.train_step(X, idx, y, step), b.train_step(X, np.tile(idx, (m, 1)), y, step))
    for i in range(m):
        np.testing.assert_array_equal(a.get_params(i, 0)[0], b.get_params(i, 0)[0])
    with pytest.raises(ValueError):
        b.train_step(X, np.zeros((m + 1, 4), dtype=np.int32), y, 3)


def _zero_head(pack, i):
    L = int(pack.depth[i])
    W, b = pack.get_params(i, L)
    pack.set_params(i, L, np.zeros_like(W), np.zeros_like(b))


def test_loss_closed_forms(orc):
    d_in, B = 4, 16
    X, yc = _make_data("multiclass", B, d_in, 10, seed=0)
    idx = np.arange(B, dtype=np.int32)
    # multiclass: all-zero logits give CE = ln C
    pc = orc.OraclePack(d_in, 10, "multiclass", [2], [16], [0.2], [1e-3], [0.0], seed=1)
    _zero_head(pc, 0)
    assert abs(pc.train_step(X, idx, yc, 0, update=False)[0] - np.log(10)) < 1e-15
    # binary: zero logit gives BCE = ln 2
    _, yb = _make_data("binary", B, d_in, 1, seed=1)
    pb = orc.OraclePack(d_in, 1, "binary", [1], [16], [0.0], [1e-3], [0.0], seed=1)
    _zero_head(pb, 0)
    assert abs(pb.train_step(X, idx, yb, 0, update=False)[0] - np.log(2)) < 1e-15
    # regression: zero output gives MSE = mean y^2
    _, yr = _make_data("regression", B, d_in, 1, seed=2)
    pr = orc.OraclePack(d_in, 1, "regression", [3], [16], [0.1], [1e-3], [0.0], seed=1)
    _zero_head(pr, 0)
    want = np.mean(yr.astype(np.float64) ** 2)
    assert abs(pr.train_step(X, idx, yr, 0, update=False)[0] - want) < 1e-14
    # with zero head the logits' gradient reaches no hidden layer
    gW, gb = pr.get_grads(0, 0)
    assert np.all(gW == 0) and np.all(gb == 0)


@pytest.mark.parametrize("task,d_out", [("binary", 1), ("multiclass", 6), ("regression", 1)])
def test_predict_matches_torch_eval(orc, task, d_out):
    m, d_in = 3, 7
    hp = random_pack(m, d_in, d_out, seed=5)
    pack = orc.OraclePack(d_in, d_out, task, hp["depth"], hp["width"], hp["dropout"], hp["lr"],
                          hp["wd"], seed=3)
    X, _ = _make_data(task, 30, d_in, d_out, seed=4)
    out = pack.predict(X)
    for i in range(m):
        h = torch.tensor(X, dtype=torch.float64)
        for l in range(int(hp["depth"][i])):
            W, b = pack.get_params(i, l)
            h = F.relu(F.linear(h, torch.tensor(W), torch.tensor(b)))   # eval mode: no dropout
        W, b = pack.get_params(i, int(hp["depth"][i]))
        z = F.linear(h, torch.tensor(W), torch.tensor(b))
        ref = torch.softmax(z, 1) if task == "multiclass" else (torch.sigmoid(z) if task == "binary" else z)
        assert _rel(out[i], ref.numpy()) < 1e-12


def test_inactive_members_are_frozen(orc):
    m, d_in = 3, 5
    hp = random_pack(m, d_in, 1, seed=8)
    pack = orc.OraclePack(d_in, 1, "regression", hp["depth"], hp["width"], hp["dropout"], hp["lr"],
                          hp["wd"], seed=4)
    X, y = _make_data("regression", 20, d_in, 1, seed=5)
    idx = np.arange(20, dtype=np.int32)
    pack.train_step(X, idx, y, 0)
    before = pack.get_params(1, 0)
    pack.set_active([1, 0, 1])
    loss = pack.train_step(X, idx, y, 1)
    assert np.isnan(loss[1]) and np.isfinite(loss[0]) and np.isfinite(loss[2])
    after = pack.get_params(1, 0)
    np.testing.assert_array_equal(before[0], after[0])
    assert pack.member_steps(1) == 1 and pack.member_steps(0) == 2


def test_rejects_bad_configs(orc):
    with pytest.raises(ValueError):
        orc.OraclePack(4, 1, "binary", [0], [16], [0.1], [1e-3], [0.0], seed=0)
    with pytest.raises(ValueError):
        orc.OraclePack(4, 1, "binary", [1], [16], [1.0], [1e-3], [0.0], seed=0)
    with pytest.raises(ValueError):
        orc.OraclePack(4, 3, "binary", [1], [16], [0.1], [1e-3], [0.0], seed=0)


def test_adamw_apply_matches_torch_adamw(orc):
    """The oracle's element-wise AdamW (used by parity tests on the GPU's own
    gradients) against torch.optim.AdamW in fp64, five steps with moments
    carried, and the pack's own update equals it on the pack's gradients."""
    rng = np.random.default_rng(3)
    p0 = rng.standard_normal(257)
    lr, wd = 2.5e-3, 3e-2
    tp = torch.tensor(p0.copy(), requires_grad=True)
    opt = torch.optim.AdamW([tp], lr=lr, betas=(0.9, 0.999), eps=1e-8, weight_decay=wd)
    p, m, v = p0.copy(), None, None
    for t in range(1, 6):
        g = rng.standard_normal(257) * 10.0 ** rng.uniform(-6, 0, 257)
        tp.grad = torch.tensor(g)
        opt.step()
        p, m, v = orc.adamw_apply(p, g, t, lr, wd, m, v)
        assert _rel(p, tp.detach().numpy()) < 1e-12

    hp = random_pack(2, 6, 1, seed=12)
    pack = orc.OraclePack(6, 1, "regression", hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"],
                          seed=4)
    X, y = _make_data("regression", 40, 6, 1, seed=6)
    before = {(i, l): pack.get_params(i, l) for i in range(2) for l in range(int(hp["depth"][i]) + 1)}
    pack.train_step(X, np.arange(40, dtype=np.int32), y, 0)
    for (i, l), (W0, b0) in before.items():
        gW, gb = pack.get_grads(i, l)
        W1, b1 = pack.get_params(i, l)
        pW, _, _ = orc.adamw_apply(W0, gW, 1, float(hp["lr"][i]), float(hp["wd"][i]))
        pb, _, _ = orc.adamw_apply(b0, gb, 1, float(hp["lr"][i]), float(hp["wd"][i]))
        np.testing.assert_array_equal(pW, W1.ravel())
        np.testing.assert_array_equal(pb, b1)
