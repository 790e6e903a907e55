"""Periodic feature embeddings on the GPU (App. "Feature Embeddings") against
the oracle's (pinned in tests/test_oracle_emb.py by finite differences and by
reduction to a plain pack).

Bars as in tests/test_gpu_parity.py (rules in tests/parity.py): floats
within 1e-4 (fp32 mode) and 2e-2 (bf16 mode) of the exact fp64 oracle, with
the oracle's bf16-storage model (E and dE stored in bf16 as on the GPU)
showing where bf16 storage itself is further than that and as a second
comparison; initial values bit-exact.  The embedding parameters' gradients
are compared like the other gradients: elementwise, or norm-wise for a
member with a first-layer decision flipped at an oracle near-tie.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

import oracle  # noqa: E402
from workloads import random_pack, sample_emb  # noqa: E402
from parity import TOL, Oracles, compare_params, compare_step, rel_err  # noqa: E402
from test_gpu_parity import _check_predictions, make_data, to_dev  # noqa: E402
from test_gpu_online import ens_mean  # noqa: E402

DEV = "cuda"


@pytest.fixture(scope="module")
def tp():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_05380_gb300 import build
    build.build()
    import paper_2607_05380_gb300 as tpm
    tpm.load_library()
    return tpm


def emb_pair(tp, task, d_in, d_out, hp, em, prec, max_batch, seed=2):
    pk = tp.Pack(d_in, d_out, task, hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"],
                 max_batch=max_batch, seed=seed, precision=prec, d_emb=em["d_emb"], freq=em["freq"])
    orc = Oracles(prec, d_in, d_out, task, hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"],
                  seed=seed, d_emb=em["d_emb"], freq=em["freq"].astype(np.float64))
    return pk, orc


def randomise_emb(pk, orc, em, d_in, seed):
    """Non-zero b, alpha and beta (from the zero start the cosine parts get
    no gradient), the same fp32 values on both sides."""
    rng = np.random.default_rng(seed)
    for i, d in enumerate(em["d_emb"]):
        d = int(d)
        w, _, _, _ = orc.emb(i)
        parts = [w, rng.uniform(-np.pi, np.pi, (d_in, d - 1)), rng.standard_normal((d_in, d)) * 0.7,
                 rng.standard_normal((d_in, d)) * 0.2]
        parts = [np.asarray(p, dtype=np.float32) for p in parts]
        pk.set_emb(i, *parts)
        orc.set_emb(i, *[p.astype(np.float64) for p in parts])


def emb_grads(pk, orc):
    """compare_step's callback: (gpu, exact, bf16 storage) embedding
    gradients [w, b, alpha, beta] of GPU member i / oracle member oi."""
    def f(i, oi):
        gx = orc.ex.emb(oi, grads=True)
        gb = orc.bst.emb(oi, grads=True) if orc.bst is not None else gx
        return [(g, x, b) for g, x, b in zip(pk.emb(i, grads=True), gx, gb) if g.size]
    return f


def emb_params(pk, orc):
    """compare_params' callback: the embedding parameters."""
    def f(i, oi):
        px = orc.ex.emb(oi)
        pb = orc.bst.emb(oi) if orc.bst is not None else px
        return [("emb_" + n, g, x, b) for n, g, x, b in zip(("w", "b", "alpha", "beta"), pk.emb(i), px, pb)
                if g.size]
    return f


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_emb_init_bit_exact(tp, prec):
    """The first layer's init over fan-in d_in d_emb, and the embedding
    parameters as given (w = freq, b = alpha = beta = 0)."""
    d_in, d_out, m = 11, 3, 4
    hp = random_pack(m, d_in, d_out, seed=3)
    em = sample_emb(m, d_in, seed=3)
    pk, orc = emb_pair(tp, "multiclass", d_in, d_out, hp, em, prec, 64)
    off = 0
    for i in range(m):
        d = int(em["d_emb"][i])
        for l in range(int(hp["depth"][i]) + 1):
            W, b = pk.get_params(i, l)
            Wo, bo = orc.get_params(i, l)
            np.testing.assert_array_equal(W, Wo.astype(np.float32))
            np.testing.assert_array_equal(b, bo.astype(np.float32))
        w, bb, a, be = pk.emb(i)
        np.testing.assert_array_equal(w.ravel(), em["freq"][off:off + d_in * (d - 1)])
        off += d_in * (d - 1)
        assert not bb.any() and not a.any() and not be.any()


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
@pytest.mark.parametrize("task,d_out", [("binary", 1), ("multiclass", 7), ("regression", 1)])
@pytest.mark.parametrize("B", [200, 1])
def test_emb_one_step(tp, prec, task, d_out, B):
    """Logits, losses, every gradient (weights, biases, embeddings) of one
    step; d_emb from the paper's range 8..32 plus 1 and 3 (the x component
    alone; an input width that is not a multiple of 8), several 128-row
    tiles and a ragged tail (B = 200), and B = 1."""
    d_in, m = 13, 6
    hp = random_pack(m, d_in, d_out, seed=80 + d_out, width=(16, 128, 16), depth=(1, 3))
    em = sample_emb_fixed(m, d_in, [1, 3, 8, 16, 24, 32], seed=4)
    pk, orc = emb_pair(tp, task, d_in, d_out, hp, em, prec, 256)
    randomise_emb(pk, orc, em, d_in, seed=5)
    X, y = make_data(task, 400, d_in, d_out, 1)
    idx = np.random.default_rng(2).choice(400, B, replace=False).astype(np.int32)
    Xd, yd, idxd = to_dev(X, y, idx)
    loss = torch.zeros(m, dtype=torch.float32, device=DEV)
    pk.forward_backward(Xd, idxd, yd, 5, loss)
    orc.train_step(X, idx, y, 5, update=False)
    problems = compare_step(pk, orc, hp, prec, loss.cpu().numpy(), emb_grads=emb_grads(pk, orc))
    assert not problems, problems


def sample_emb_fixed(m, d_in, d_emb, seed):
    """Frequencies ~ N(0, 1) for given embedding sizes."""
    rng = np.random.default_rng([seed, 11])
    freq = np.concatenate([rng.standard_normal(d_in * (int(d) - 1)) for d in d_emb] + [np.zeros(0)])
    return dict(d_emb=np.asarray(d_emb, dtype=np.int32), freq=freq.astype(np.float32))


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_emb_stacked_one_step(tp, prec):
    """A batch per member (idx [m, B]): each member's embeddings read its own
    rows."""
    d_in, m, B, d_out = 13, 5, 160, 4
    hp = random_pack(m, d_in, d_out, seed=91, width=(16, 96, 16), depth=(1, 3))
    em = sample_emb(m, d_in, seed=6)
    pk, orc = emb_pair(tp, "multiclass", d_in, d_out, hp, em, prec, 256)
    randomise_emb(pk, orc, em, d_in, seed=7)
    X, y = make_data("multiclass", 400, d_in, d_out, 2)
    rng = np.random.default_rng(3)
    idx = np.stack([rng.choice(400, B, replace=False) for _ in range(m)]).astype(np.int32)
    Xd, yd, idxd = to_dev(X, y, idx)
    loss = torch.zeros(m, dtype=torch.float32, device=DEV)
    pk.forward_backward(Xd, idxd, yd, 2, loss)
    orc.train_step(X, idx, y, 2, update=False)
    problems = compare_step(pk, orc, hp, prec, loss.cpu().numpy(), emb_grads=emb_grads(pk, orc))
    assert not problems, problems


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_emb_eight_steps(tp, prec):
    """AdamW on every parameter including the embeddings over eight steps
    from the paper's zero start of b, alpha and beta (graph replay after the
    first step; a stacked step in the middle).

    bf16: against the exact oracle by the rule of tests/parity.py.  Adam's
    first updates are about lr times the sign of the gradient, so a
    parameter that starts at zero (b, alpha, beta) and a gradient within
    bf16 rounding of zero move by +-lr on one side and -+lr on the other:
    the diagnostic comparison with the bf16-storage oracle then allows a
    tensor that misses its elementwise bar to be no further from that oracle
    than three times its distance from the exact one (norm-wise)."""
    d_in, m, B, d_out = 9, 6, 192, 3
    hp = random_pack(m, d_in, d_out, seed=93, width=(16, 96, 16), depth=(1, 3))
    em = sample_emb(m, d_in, seed=8, sigma=(0.1, 1.0))
    pk, orc = emb_pair(tp, "multiclass", d_in, d_out, hp, em, prec, 256)
    X, y = make_data("multiclass", 600, d_in, d_out, 3)
    Xd, yd = to_dev(X, y)
    rng = np.random.default_rng(5)
    loss = torch.zeros(m, dtype=torch.float32, device=DEV)
    margin = np.full(m, np.inf)
    for step in range(8):
        if step == 4:
            idx = np.stack([rng.choice(600, B, replace=False) for _ in range(m)]).astype(np.int32)
        else:
            idx = rng.choice(600, B, replace=False).astype(np.int32)
        (idxd,) = to_dev(idx)
        pk.train_step(Xd, idxd, yd, step, loss)
        lo = orc.train_step(X, idx, y, step)
        margin = np.minimum(margin, [orc.margin(i) for i in range(m)])
        lg = loss.cpu().numpy()
        for i in range(m):
            bar = TOL[prec] if (prec == "bf16" or margin[i] >= 1e-5) else TOL["bf16"]
            assert abs(lg[i] - lo[i]) <= bar * max(1.0, abs(lo[i])), (step, i, lg[i], lo[i])
    errs, problems, relaxed = compare_params(pk, orc, hp, prec, margin=margin, extra=emb_params(pk, orc),
                                             diag_ratio=3.0)
    assert not problems and len(relaxed) <= m // 3, (problems, errs, relaxed, margin)


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_emb_muon_one_step(tp, prec):
    """Muon on the first layer's [width, d_in d_emb] matrix (AdamW on the
    embeddings): parameters after one step (fp32 against the oracle; bf16
    by the bf16 rule against the exact oracle).  The bf16 kernel stores U and
    applies 1 / |U|_F in fp32 inside the first Newton-Schulz products, while
    the oracle's bf16-storage model rounds U / |U|_F: two bf16 roundings of
    the same iteration, each within d of the exact result, so the diagnostic
    comparison with the model is norm-wise within 2 d (triangle inequality)
    where it misses 2e-2 elementwise."""
    d_in, m, B, d_out = 7, 4, 160, 3
    hp = random_pack(m, d_in, d_out, seed=95, width=(16, 96, 16), depth=(1, 2), dropout=(0.0, 0.0))
    em = sample_emb(m, d_in, seed=9)
    pk, orc = emb_pair(tp, "multiclass", d_in, d_out, hp, em, prec, 256)
    randomise_emb(pk, orc, em, d_in, seed=10)
    lr_m = np.full(m, 0.02, dtype=np.float32)
    pk.set_muon(lr_m)
    orc.set_muon(lr_m.astype(np.float64))
    X, y = make_data("multiclass", 300, d_in, d_out, 4)
    idx = np.random.default_rng(6).choice(300, B, replace=False).astype(np.int32)
    Xd, yd, idxd = to_dev(X, y, idx)
    pk.train_step(Xd, idxd, yd, 0)
    orc.train_step(X, idx, y, 0)
    errs, problems, relaxed = compare_params(pk, orc, hp, prec, extra=emb_params(pk, orc), diag_ratio=2.0)
    assert not problems and not relaxed, (problems, errs)


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_emb_predict(tp, prec):
    """Predictions (fp32: chunks of max_batch rows, ragged tail; bf16: one
    chunk) against the oracle."""
    d_in, d_out, m = 10, 5, 5
    hp = random_pack(m, d_in, d_out, seed=97, width=(16, 96, 16))
    em = sample_emb(m, d_in, seed=11)
    pk, orc = emb_pair(tp, "multiclass", d_in, d_out, hp, em, prec, 128)
    randomise_emb(pk, orc, em, d_in, seed=12)
    X, _ = make_data("multiclass", 333, d_in, d_out, 5)
    (Xd,) = to_dev(X)
    out = pk.predict(Xd).cpu().numpy()
    _check_predictions(out, orc, X, prec)


def test_emb_predict_chunk_cap(tp):
    """Wide embeddings (4 members x 1024 features x d_emb 16): the chunk's
    embedding matrices would pass 1 GiB at 8192 rows, so bf16 prediction
    runs in smaller chunks (8064 rows).  Rows of the second chunk predict
    the same alone (bit-exact), and sampled rows of both chunks match the
    oracle."""
    d_in, d_out, m, N = 1024, 2, 4, 8200
    hp = random_pack(m, d_in, d_out, seed=99, width=(16, 48, 16), depth=(1, 2))
    em = sample_emb_fixed(m, d_in, [16] * m, seed=13)
    pk, orc = emb_pair(tp, "multiclass", d_in, d_out, hp, em, "bf16", 64)
    randomise_emb(pk, orc, em, d_in, seed=14)
    X, _ = make_data("multiclass", N, d_in, d_out, 6)
    (Xd,) = to_dev(X)
    full = pk.predict(Xd).cpu().numpy()
    np.testing.assert_array_equal(pk.predict(Xd[8064:].contiguous()).cpu().numpy(), full[:, 8064:])
    rows = np.r_[0:40, 8040:8100, 8160:8200]
    _check_predictions(np.ascontiguousarray(full[:, rows]), orc, X[rows], "bf16")


def test_emb_online_ensemble(tp):
    """The online ensemble of a pack with embeddings: its prediction is the
    fp64 mean of the pack's predictions of the selected members at the
    epoch they were recorded (the ensemble pack is rebuilt with the same
    embedding sizes from the snapshots)."""
    d_in, d_out, m, n_val = 8, 3, 6, 300
    hp = random_pack(m, d_in, d_out, seed=101, width=(16, 64, 16))
    em = sample_emb(m, d_in, seed=15)
    pk, _ = emb_pair(tp, "multiclass", d_in, d_out, hp, em, "bf16", 128)
    X, y = make_data("multiclass", 800, d_in, d_out, 7)
    Xd, yd = to_dev(X, y)
    Xv, yv = Xd[:n_val].contiguous(), yd[:n_val].contiguous()
    Xt = Xd[n_val:].contiguous()
    on = tp.OnlineEnsemble(pk, n_val, score="loss", m_ens=4, p_base=4, p_ens=4)
    rec = {}
    rng = np.random.default_rng(8)
    for ep in range(1, 4):   # the online ensemble numbers epochs from 1
        for s in range(4):
            idx = (n_val + rng.choice(500, 128, replace=False)).astype(np.int32)
            (idxd,) = to_dev(idx)
            pk.train_step(Xd, idxd, yd, ep * 4 + s)
        pt = pk.predict(Xt).cpu().numpy()
        for i in range(m):
            rec[(i, ep)] = pt[i]
        on.epoch(Xv, yv)
    mem, eps, _ = on.ensemble("best")
    got = on.predict(Xt).cpu().numpy()
    assert np.array_equal(got, ens_mean([rec[(int(a), int(b))] for a, b in zip(mem, eps)]))


def test_emb_full_size_sampled_members(tp):
    """The medium workload with embeddings as `bench.py --emb` runs it (the
    whole pack of 32 members, batch 512, bf16, the embedding sizes and
    frequencies the bench samples): for the cheapest member of each depth
    (embedding parameters set to random values on both sides: from the
    paper's zero start E is zero), losses, logits, every gradient and the
    embedding gradients against the oracle run on those members alone
    (members are independent, Sec. 3.6)."""
    from workloads import SEED_HP, SEED_INIT, WORKLOADS, make_data as wl_data, sample_hparams
    from test_gpu_parity import _sample_members
    wl = WORKLOADS["medium"]
    hp = sample_hparams(wl, seed=SEED_HP)
    em = sample_emb(wl.m, wl.d_in, seed=SEED_HP + 200)
    B = wl.batch
    d = wl_data(wl, device="cpu", n_train=3 * B, n_val=0)
    X, y = d["X_train"].numpy(), d["y_train"].numpy()
    Xd, yd = to_dev(X, y)
    idx = np.random.default_rng(3).permutation(3 * B)[:B].astype(np.int32)
    (idxd,) = to_dev(idx)
    sample = _sample_members(wl, hp)
    sub = {k: v[sample] for k, v in hp.items()}
    starts = np.concatenate([[0], np.cumsum(wl.d_in * (em["d_emb"] - 1))])
    freq_sub = np.concatenate([em["freq"][starts[i]:starts[i + 1]] for i in sample])
    pk = tp.Pack(wl.d_in, wl.d_out, wl.task, hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"],
                 max_batch=B, seed=SEED_INIT, precision="bf16", d_emb=em["d_emb"], freq=em["freq"])
    orc = Oracles("bf16", wl.d_in, wl.d_out, wl.task, sub["depth"], sub["width"], sub["dropout"], sub["lr"],
                  sub["wd"], seed=SEED_INIT, member_id=sample, d_emb=em["d_emb"][sample],
                  freq=freq_sub.astype(np.float64))
    rng = np.random.default_rng(21)
    for oi, i in enumerate(sample):
        dm = int(em["d_emb"][i])
        parts = [np.asarray(p, dtype=np.float32) for p in (
            pk.emb(i)[0], rng.uniform(-np.pi, np.pi, (wl.d_in, dm - 1)), rng.standard_normal((wl.d_in, dm)) * 0.7,
            rng.standard_normal((wl.d_in, dm)) * 0.2)]
        pk.set_emb(i, *parts)
        orc.set_emb(oi, *[p.astype(np.float64) for p in parts])
    loss = torch.zeros(wl.m, dtype=torch.float32, device=DEV)
    pk.forward_backward(Xd, idxd, yd, 0, loss)
    orc.train_step(X, idx, y, 0, update=False)
    problems = compare_step(pk, orc, hp, "bf16", loss.cpu().numpy(), members=sample, emb_grads=emb_grads(pk, orc))
    assert not problems, problems


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
@pytest.mark.parametrize("wd_on_bias", [False, True])
def test_emb_weight_decay_follows_the_bias_flag(tp, prec, wd_on_bias):
    """From the paper's zero start (alpha = 0) w and b get a zero gradient:
    with wd_on_bias off one AdamW step leaves w bit-identical, with it on w
    shrinks by lr wd w (fp32 arithmetic); b stays zero; alpha moves."""
    d_in, d_out, m = 6, 3, 3
    hp = random_pack(m, d_in, d_out, seed=103, width=(16, 64, 16))
    em = sample_emb(m, d_in, seed=16)
    pk = tp.Pack(d_in, d_out, "multiclass", hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"],
                 max_batch=128, seed=2, precision=prec, wd_on_bias=wd_on_bias, d_emb=em["d_emb"], freq=em["freq"])
    X, y = make_data("multiclass", 200, d_in, d_out, 9)
    Xd, yd = to_dev(X, y)
    before = [pk.emb(i) for i in range(m)]
    (idxd,) = to_dev(np.arange(128, dtype=np.int32))
    pk.train_step(Xd, idxd, yd, 0)
    for i in range(m):
        w0 = before[i][0]
        w1, b1, a1, _ = pk.emb(i)
        if wd_on_bias:
            expect = w0.astype(np.float64) * (1.0 - float(np.float32(hp["lr"][i])) * float(np.float32(hp["wd"][i])))
            np.testing.assert_allclose(w1, expect, rtol=1e-6, atol=0)
        else:
            np.testing.assert_array_equal(w1, w0)
        assert not b1.any() and np.abs(a1).max() > 0


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_emb_maximum_size(tp, prec):
    """The largest embedding the library takes (d_emb = 64) on 40 features:
    a first layer of 2560 inputs (40 K blocks), next to a d_emb = 2 member;
    one step's logits, losses and every gradient against the oracle."""
    d_in, d_out, m = 40, 4, 2
    hp = random_pack(m, d_in, d_out, seed=107, width=(32, 96, 16), depth=(1, 2))
    em = sample_emb_fixed(m, d_in, [64, 2], seed=17)
    pk, orc = emb_pair(tp, "multiclass", d_in, d_out, hp, em, prec, 256)
    randomise_emb(pk, orc, em, d_in, seed=18)
    X, y = make_data("multiclass", 300, d_in, d_out, 11)
    idx = np.random.default_rng(12).choice(300, 130, replace=False).astype(np.int32)
    Xd, yd, idxd = to_dev(X, y, idx)
    loss = torch.zeros(m, dtype=torch.float32, device=DEV)
    pk.forward_backward(Xd, idxd, yd, 3, loss)
    orc.train_step(X, idx, y, 3, update=False)
    problems = compare_step(pk, orc, hp, prec, loss.cpu().numpy(), emb_grads=emb_grads(pk, orc))
    assert not problems, problems
