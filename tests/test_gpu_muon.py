"""Muon on the GPU (hidden-layer weights; Sec. 3.4, App. F.1) against the
oracle's Muon (pinned against torch.optim.Muon in tests/test_oracle_muon.py).

Bars: fp32 mode (the iteration on CUDA cores in fp32): the Newton-Schulz
direction of every hidden layer after a step within 1e-4 of the oracle's,
relative to max(|o|, rms(o)) as in the other parity tests.  bf16 mode (the
products on the tensor cores with X, A and B stored in bf16): the direction
computed from the GPU's own gradient within twice the error that the oracle's
bf16 rounding model of the same iteration makes against the exact one (norm-
wise; see the test).  Parameters after one step within 1e-4 of the exact
oracle (fp32); in bf16 against the exact oracle by the rule of
tests/parity.py (2e-2, or twice the oracle's own bf16-storage distance from
the exact result), and within 2e-2 of the bf16-storage oracle as a second
comparison.  After eight steps within 1e-4 (fp32), and in bf16 by the same
exact-oracle rule, with the bf16-storage comparison allowing three times the
distance between the bf16 and the exact oracle (see the test).
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

import oracle  # noqa: E402
from parity import Oracles, check_bf16_vs_exact  # noqa: E402
from workloads import random_pack  # noqa: E402

DEV = "cuda"
TOL = {"fp32": 1e-4, "bf16": 2e-2}


@pytest.fixture(scope="module")
def tp():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_05380_gb300 import build
    build.build()
    import paper_2607_05380_gb300 as tpm
    tpm.load_library()
    return tpm


def rel_err(got, ref):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    rms = np.sqrt(np.mean(ref ** 2))
    return float(np.max(np.abs(got - ref) / np.maximum(np.abs(ref), rms if rms > 0 else 1e-30)))


def make(tp, task, d_in, d_out, hp, prec, lr_m, max_batch=256):
    pk = tp.Pack(d_in, d_out, task, hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"],
                 max_batch=max_batch, seed=2, precision=prec)
    orc = Oracles(prec, d_in, d_out, task, hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"], seed=2)
    pk.set_muon(lr_m)
    orc.set_muon(lr_m.astype(np.float64))
    return pk, orc


def data(task, n, d_in, d_out, seed):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((n, d_in)).astype(np.float32)
    if task == "regression":
        y = rng.standard_normal(n).astype(np.float32)
    else:
        y = rng.integers(0, max(d_out, 2), n).astype(np.int32)
    return X, y


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
@pytest.mark.parametrize("task,d_out", [("multiclass", 5), ("regression", 1)])
def test_muon_direction_one_step(tp, prec, task, d_out):
    """Hidden widths 16..160 (tiles split in columns, ragged r), d_in = 37
    (layer 1 wide or tall, so X is taken transposed for the wider members)."""
    d_in, m, B = 37, 6, 200
    hp = random_pack(m, d_in, d_out, seed=60 + d_out, width=(16, 160, 16), depth=(1, 3))
    lr_m = np.exp(np.random.default_rng(1).uniform(np.log(1e-3), np.log(5e-2), m)).astype(np.float32)
    pk, orc = make(tp, task, d_in, d_out, hp, prec, lr_m)
    X, y = data(task, 400, d_in, d_out, 1)
    idx = np.random.default_rng(2).choice(400, B, replace=False).astype(np.int32)
    Xd, yd, idxd = (torch.from_numpy(a).to(DEV) for a in (X, y, idx))
    pk.train_step(Xd, idxd, yd, 3)
    orc.train_step(X, idx, y, 3)
    errs = {}
    for i in range(m):
        for l in range(int(hp["depth"][i])):
            O = pk.muon_dir(i, l)
            if prec == "fp32":
                errs[(i, l, "dir")] = rel_err(O, orc.muon_dir(i, l))
            else:
                # bf16: the orthogonalisation of the GPU's own gradient (the first
                # step's X0 is G / |G|) against the exact iteration, allowed twice
                # the error of the oracle's bf16 rounding model of the same
                # iteration -- the direction of a near-singular spectrum is
                # sensitive to one-ulp differences, so elementwise comparison
                # with the oracle (whose gradient differs at the bf16 level) is
                # not a meaningful bar
                G = pk.get_grads(i, l)[0].astype(np.float64)
                O_ref = oracle.newton_schulz(G)
                e_orc = np.linalg.norm(oracle.newton_schulz(G, bf16=True) - O_ref) / np.linalg.norm(O_ref)
                e_gpu = np.linalg.norm(O - O_ref) / np.linalg.norm(O_ref)
                errs[(i, l, "dir")] = 0.0 if e_gpu <= max(2.0 * e_orc, 5e-3) else e_gpu
        for l in range(int(hp["depth"][i]) + 1):
            W, b = pk.get_params(i, l)
            if prec == "fp32":
                Wo, bo = orc.ex.get_params(i, l)
                errs[(i, l, "W")] = max(rel_err(W, Wo), rel_err(b, bo))
            else:
                Wo, bo = orc.bst.get_params(i, l)
                errs[(i, l, "W")] = max(rel_err(W, Wo), rel_err(b, bo))
                p = []
                for g_, ob, ox in zip((W, b), (Wo, bo), orc.ex.get_params(i, l)):
                    check_bf16_vs_exact("params", g_, ob, ox, p, (i, l))
                if p:
                    errs[(i, l, "vs exact")] = 1.0
    bad = {k: e for k, e in errs.items() if e > TOL[prec]}
    assert not bad, bad


@pytest.mark.parametrize("prec", ["fp32", "bf16"])
def test_muon_eight_steps(tp, prec):
    """Momentum across steps, graph replay after the first step."""
    d_in, m, B, d_out = 24, 5, 192, 3
    hp = random_pack(m, d_in, d_out, seed=71, width=(32, 128, 16), depth=(1, 3))
    lr_m = np.full(m, 0.02, dtype=np.float32)
    pk, orc = make(tp, "multiclass", d_in, d_out, hp, prec, lr_m)
    # bf16: the exact-arithmetic oracle beside the bf16-storage one measures
    # how far bf16 storage alone moves the trajectory
    X, y = data("multiclass", 600, d_in, d_out, 3)
    Xd, yd = (torch.from_numpy(a).to(DEV) for a in (X, y))
    rng = np.random.default_rng(5)
    loss = torch.zeros(m, dtype=torch.float32, device=DEV)
    for step in range(8):
        idx = rng.choice(600, B, replace=False).astype(np.int32)
        pk.train_step(Xd, torch.from_numpy(idx).to(DEV), yd, step, loss)
        lo = orc.train_step(X, idx, y, step)
        lg = loss.cpu().numpy()
        for i in range(m):
            assert abs(lg[i] - lo[i]) <= TOL["bf16"] * max(1.0, abs(lo[i])), (step, i, lg[i], lo[i])
    errs = {}
    for i in range(m):
        for l in range(int(hp["depth"][i]) + 1):
            W, b = pk.get_params(i, l)
            if prec == "fp32":
                Wo, bo = orc.ex.get_params(i, l)
                errs[(i, l)] = max(rel_err(W, Wo), rel_err(b, bo))
            else:
                Wo, bo = orc.bst.get_params(i, l)
                exact = orc.ex
                p = []
                for g_, ob, ox in zip((W, b), (Wo, bo), exact.get_params(i, l)):
                    check_bf16_vs_exact("params", g_, ob, ox, p, (i, l))
                if p:
                    errs[(i, l, "vs exact")] = 1.0
                # the bf16 Newton-Schulz direction of a near-singular spectrum
                # moves by a few per cent with one-ulp changes (one-step test),
                # so two bf16 trajectories drift apart; bar: the GPU's distance
                # from the bf16 oracle within three times the distance between
                # the bf16 oracle and the exact one (norm-wise per tensor)
                We, be = exact.get_params(i, l)
                for g_, o_, e_ in ((W, Wo, We), (b, bo, be)):
                    d_gpu = np.linalg.norm(g_ - o_) / max(np.linalg.norm(o_), 1e-30)
                    d_ref = np.linalg.norm(o_ - e_) / max(np.linalg.norm(e_), 1e-30)
                    errs[(i, l, len(g_.shape))] = 0.0 if d_gpu <= max(3.0 * d_ref, 1e-3) else d_gpu
    bad = {k: e for k, e in errs.items() if e > TOL[prec]}
    assert not bad, bad


def test_muon_argument_checks(tp):
    hp = random_pack(2, 8, 1, seed=3)
    pk = tp.Pack(8, 1, "regression", hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"], max_batch=64)
    with pytest.raises(tp.TabpackError):
        pk.set_muon(np.array([0.01, -1.0], dtype=np.float32))
    with pytest.raises(tp.TabpackError):
        pk.set_muon(np.array([0.01, 0.01], dtype=np.float32), momentum=1.0)
    with pytest.raises(tp.TabpackError):
        pk.muon_dir(0, 0)   # Muon not on yet


def test_muon_full_size_sampled_members(tp):
    """The medium workload with Muon as `bench.py --muon` runs it (the whole
    pack, batch 512, bf16, the bench's per-member Muon learning rates): one
    step; for the cheapest member of each depth, the Newton-Schulz direction
    of every hidden layer from the GPU's own gradient within twice the error
    of the oracle's bf16 model of the iteration (norm-wise, against the exact
    iteration), and the parameters after the step within 2e-2 elementwise of
    the bf16 oracle run on those members alone, or no further from it than
    three times the distance between the bf16 and the exact oracle."""
    import math
    from workloads import SEED_HP, SEED_INIT, WORKLOADS, make_data as wl_data, sample_hparams
    from test_gpu_parity import _sample_members
    wl = WORKLOADS["medium"]
    hp = sample_hparams(wl, seed=SEED_HP)
    rng_m = np.random.default_rng(SEED_HP + 100)
    lr_m = np.exp(rng_m.uniform(math.log(1e-3), math.log(1e-1), wl.m)).astype(np.float32)
    B = wl.batch
    d = wl_data(wl, device="cpu", n_train=3 * B, n_val=0)
    X, y = d["X_train"].numpy(), d["y_train"].numpy()
    Xd, yd = (torch.from_numpy(a).to(DEV) for a in (X, y))
    idx = np.random.default_rng(3).permutation(3 * B)[:B].astype(np.int32)
    sample = _sample_members(wl, hp)
    sub = {k: v[sample] for k, v in hp.items()}
    pk = tp.Pack(wl.d_in, wl.d_out, wl.task, hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"],
                 max_batch=B, seed=SEED_INIT, precision="bf16")
    pk.set_muon(lr_m)
    orcs = []
    for bf in (True, False):
        o = oracle.OraclePack(wl.d_in, wl.d_out, wl.task, sub["depth"], sub["width"], sub["dropout"], sub["lr"],
                              sub["wd"], seed=SEED_INIT, bf16_storage=bf, member_id=sample)
        o.set_muon(lr_m[sample].astype(np.float64))
        o.train_step(X, idx, y, 0)
        orcs.append(o)
    orc, exact = orcs
    pk.train_step(Xd, torch.from_numpy(idx).to(DEV), yd, 0)
    errs = {}
    for oi, i in enumerate(sample):
        for l in range(int(hp["depth"][i])):
            G = pk.get_grads(i, l)[0].astype(np.float64)
            O_ref = oracle.newton_schulz(G)
            e_orc = np.linalg.norm(oracle.newton_schulz(G, bf16=True) - O_ref) / np.linalg.norm(O_ref)
            e_gpu = np.linalg.norm(pk.muon_dir(i, l) - O_ref) / np.linalg.norm(O_ref)
            errs[(i, l, "dir")] = 0.0 if e_gpu <= max(2.0 * e_orc, 5e-3) else e_gpu
        for l in range(int(hp["depth"][i]) + 1):
            for g_, o_, e_ in zip(pk.get_params(i, l), orc.get_params(oi, l), exact.get_params(oi, l)):
                p = []
                check_bf16_vs_exact("params", g_, o_, e_, p, (i, l))
                if p:
                    errs[(i, l, "vs exact")] = 1.0
                e = rel_err(g_, o_)
                if e > TOL["bf16"]:
                    d_gpu = np.linalg.norm(g_ - o_) / max(np.linalg.norm(o_), 1e-30)
                    d_ref = np.linalg.norm(o_ - e_) / max(np.linalg.norm(e_), 1e-30)
                    e = 0.0 if d_gpu <= max(3.0 * d_ref, 1e-3) else e
                errs[(i, l, len(g_.shape))] = max(errs.get((i, l, len(g_.shape)), 0.0), e)
    bad = {k: e for k, e in errs.items() if e > TOL["bf16"]}
    assert not bad, bad


@pytest.mark.parametrize("ctas", ["1", "2"])
@pytest.mark.parametrize("ns_steps", [1, 2, 3])
def test_muon_ns_steps_and_cta_pairs(tp, monkeypatch, ns_steps, ctas):
    """The single Newton-Schulz launch of bf16 mode (every iteration's three
    products, chained by per-matrix counters) for 1, 2 and 3 iterations (the
    result in either X buffer), with single CTAs and with CTA pairs. Widths
    384 and 640 leave the second CTA of a pair's last row tile without rows, so
    it waits and loads its half of B only for its partner. The tall first
    layers (384 and 640 outputs over 200 inputs) run transposed, and the middle
    member is inactive. Bar, per active member and layer: the direction from
    the GPU's own gradient within twice the error that the oracle's bf16 model
    of the same iteration makes against the exact one (norm-wise), or 5e-3."""
    monkeypatch.setenv("TP_GEMM_CTAS", ctas)
    d_in, d_out, B = 200, 4, 256
    hp = {"depth": np.array([2, 1, 2], dtype=np.int32), "width": np.array([384, 256, 640], dtype=np.int32),
          "dropout": np.array([0.0, 0.1, 0.2], dtype=np.float32), "lr": np.full(3, 1e-3, dtype=np.float32),
          "wd": np.full(3, 1e-4, dtype=np.float32)}
    pk = tp.Pack(d_in, d_out, "multiclass", hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"],
                 max_batch=B, seed=4, precision="bf16")
    pk.set_muon(np.full(3, 0.02, dtype=np.float32), ns_steps=ns_steps)
    pk.set_active(np.array([1, 0, 1], dtype=np.uint8))
    X, y = data("multiclass", 2 * B, d_in, d_out, 11)
    Xd, yd = (torch.from_numpy(a).to(DEV) for a in (X, y))
    idx = np.random.default_rng(2).permutation(2 * B)[:B].astype(np.int32)
    pk.train_step(Xd, torch.from_numpy(idx).to(DEV), yd, 0)
    errs = {}
    for i in (0, 2):
        for l in range(int(hp["depth"][i])):
            G = pk.get_grads(i, l)[0].astype(np.float64)
            O_ref = oracle.newton_schulz(G, steps=ns_steps)
            e_orc = np.linalg.norm(oracle.newton_schulz(G, steps=ns_steps, bf16=True) - O_ref) / np.linalg.norm(O_ref)
            e_gpu = np.linalg.norm(pk.muon_dir(i, l) - O_ref) / np.linalg.norm(O_ref)
            if e_gpu > max(2.0 * e_orc, 5e-3):
                errs[(i, l)] = (e_gpu, e_orc)
    assert not errs, errs
