"""Online ensemble on the GPU (Sec. 3.5 "Online ensemble", Sec. 3.6 early
stopping) against the oracle's epoch-end logic (oracle/online.py).

Each epoch the test reads the pack's validation predictions through
pack_predict (the call the online object makes on the same state, so the
values are the same) and hands them to the oracle, which forms its own pool,
selects with fp32 per-row terms (the GPU scorer's decision precision) and
applies the patience rules.  Bars: selected instances, removed members, the
stop flag and the best ensemble identical (a selection may differ only where
the oracle's best-vs-runner-up margin is a near-tie, after which the runs are
no longer comparable); scores within 1e-6 relative (per-row fp32 terms: the
device's logf and the host's may differ by an ulp, 2^-23 relative, in each
term; plus fp64 sums in another order); snapshots and the ensemble prediction bit-exact against the recorded
states and predictions.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from oracle.online import OnlineEnsemble as OracleOnline  # noqa: E402
from workloads import WORKLOADS, batch_indices, make_data, sample_hparams  # noqa: E402


@pytest.fixture(scope="module")
def tp():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_05380_gb300 import build
    build.build()
    import paper_2607_05380_gb300 as tpm
    tpm.load_library()
    return tpm


SCORE_REL = 1e-6


def near_tie(r, k):
    return r["step_gap"][k] <= 1e-6 * max(1.0, abs(r["step_best"][k]))


def diverged_at_near_tie(r, got, sc, k):
    """The GPU's and the oracle's selections first differ at step k: allowed
    only where the decision taken there was within rounding on the oracle's
    side."""
    ours = r["selected"]
    if k < len(ours) and k < len(got):          # different picks: runner-up within rounding
        return near_tie(r, k)
    if len(ours) > len(got):                    # the GPU stopped: the oracle's last addition barely improved
        return abs(r["step_best"][k] - r["step_best"][k - 1]) <= 2 * SCORE_REL * abs(r["step_best"][k - 1])
    return abs(sc - r["score"]) <= 2 * SCORE_REL * abs(r["score"])   # the oracle stopped


def ens_mean(preds):
    """The ensemble prediction as the library defines it: fp64 sum in order,
    times 1/n, rounded to fp32."""
    s = np.zeros(preds[0].shape, dtype=np.float64)
    for p in preds:
        s += p.astype(np.float64)
    return (s * (1.0 / len(preds))).astype(np.float32)


def setup(tp, wl_name, prec, m=None, n_train=None, n_val=None, lr_zero=(), seed_hp=1):
    wl = WORKLOADS[wl_name]
    data = make_data(wl, device="cuda", n_train=n_train, n_val=n_val)
    hp = sample_hparams(wl, seed=seed_hp, m=m)
    lr = hp["lr"].copy()
    for i in lr_zero:
        lr[i] = 0.0
    pk = tp.Pack(wl.d_in, wl.d_out, wl.task, hp["depth"], hp["width"], hp["dropout"], lr, hp["wd"], wl.batch,
                 precision=prec)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(11)
    X_test = torch.randn(1000, wl.d_in, generator=gen, device="cuda")
    return wl, data, pk, X_test


def run_online(tp, wl, data, pk, X_test, score, m_ens, p_base, p_ens, epochs):
    on = tp.OnlineEnsemble(pk, data["X_val"].shape[0], score, m_ens, p_base, p_ens)
    orc = OracleOnline(pk.m, wl.task, score, m_ens, p_base, p_ens)
    y_val = data["y_val"].cpu().numpy()
    n_train = data["X_train"].shape[0]
    rec_val, rec_test, rec_snap = {}, {}, {}
    step, comparable, n_epochs = 0, True, 0
    for e in range(1, epochs + 1):
        for idx in batch_indices(n_train, wl.batch, e):
            pk.train_step(data["X_train"], torch.from_numpy(idx).cuda(), data["y_train"], step)
            step += 1
        active = pk.get_active().astype(bool)
        live = pk.predict(data["X_val"]).cpu().numpy()
        live_t = pk.predict(X_test).cpu().numpy()
        for i in np.flatnonzero(active):
            rec_val[(i, e)] = live[i].copy()
            rec_test[(i, e)] = live_t[i].copy()
            rec_snap[(i, e)] = pk.snapshot(int(i)).cpu().numpy()
        prev_best = orc.member_best.copy()
        prev_ens_best = orc.best_score
        stop = on.epoch(data["X_val"], data["y_val"])
        r = orc.epoch_end(live, y_val)
        n_epochs = e
        mem, ep, sc = on.ensemble("last")
        got = [(int(a), int(b)) for a, b in zip(mem, ep)]
        if got != r["selected"]:
            k = next(k for k in range(min(len(got), len(r["selected"])) + 1)
                     if k >= len(got) or k >= len(r["selected"]) or got[k] != r["selected"][k])
            assert diverged_at_near_tie(r, got, sc, k), (e, got, r["selected"])
            comparable = False
            break
        assert sc == pytest.approx(r["score"], rel=SCORE_REL, abs=1e-12), (e, sc, r["score"])
        own, best, bad = on.members()
        for i in range(pk.m):
            if active[i]:
                assert own[i] == pytest.approx(r["own"][i], rel=SCORE_REL, abs=1e-12), (e, i)
            else:
                assert np.isnan(own[i]) and np.isnan(r["own"][i])
        # removals: identical unless an own score came within rounding of the best so far
        tie = [i for i in np.flatnonzero(active)
               if np.isfinite(prev_best[i]) and abs(r["own"][i] - prev_best[i]) <= 2 * SCORE_REL * abs(prev_best[i])
               and r["own"][i] != prev_best[i]]
        if tie:
            comparable = False      # a member's improvement decided within rounding
            break
        assert pk.get_active().astype(bool).tolist() == orc.active.tolist(), e
        assert bad.tolist() == orc.member_bad.tolist(), e
        if (np.isfinite(prev_ens_best) and r["score"] != prev_ens_best
                and abs(r["score"] - prev_ens_best) <= 2 * SCORE_REL * abs(prev_ens_best)):
            comparable = False      # ensemble improvement decided within rounding
            break
        info = on.info()
        assert info["epoch"] == e and info["n_pool"] == len(r["pool"])
        assert info["ens_bad"] == orc.ens_bad and info["best_epoch"] == orc.best_epoch
        assert bool(stop) == r["stop"] == bool(info["stop"])
        if stop:
            break
    return on, orc, rec_val, rec_test, rec_snap, comparable, n_epochs


def check_best(on, orc, data, X_test, rec_val, rec_test, rec_snap):
    mem, ep, sc = on.ensemble("best")
    best = [(int(a), int(b)) for a, b in zip(mem, ep)]
    assert best == orc.best
    assert sc == pytest.approx(orc.best_score, rel=SCORE_REL, abs=1e-12)
    for j, inst in enumerate(best):
        assert np.array_equal(on.snapshot(j).cpu().numpy(), rec_snap[inst]), inst
    pv = on.predict(data["X_val"]).cpu().numpy()
    assert np.array_equal(pv, ens_mean([rec_val[i] for i in best]))
    pt = on.predict(X_test).cpu().numpy()
    assert np.array_equal(pt, ens_mean([rec_test[i] for i in best]))


@pytest.mark.parametrize("prec,score", [("bf16", "loss"), ("fp32", "accuracy"), ("bf16", "accuracy"), ("bf16", "auc")])
def test_online_tiny_matches_oracle(tp, prec, score):
    """Tiny binary workload, 10 epochs; members 1 and 5 have lr = 0, so their
    predictions never change and p_base = 1 removes them after epoch 3."""
    wl, data, pk, X_test = setup(tp, "tiny", prec, lr_zero=(1, 5))
    on, orc, rv, rt, rs, comparable, n = run_online(tp, wl, data, pk, X_test, score, m_ens=8, p_base=1,
                                                    p_ens=4, epochs=10)
    if comparable:
        assert not orc.active[1] and not orc.active[5] and n >= 3
        check_best(on, orc, data, X_test, rv, rt, rs)


def test_online_regression_rmse(tp):
    wl, data, pk, X_test = setup(tp, "medium", "bf16", m=6, n_train=4096, n_val=2000)
    on, orc, rv, rt, rs, comparable, _ = run_online(tp, wl, data, pk, X_test, "rmse", m_ens=5, p_base=2,
                                                    p_ens=2, epochs=6)
    if comparable:
        check_best(on, orc, data, X_test, rv, rt, rs)


def test_online_multiclass_loss(tp):
    wl, data, pk, X_test = setup(tp, "large", "bf16", m=5, n_train=3072, n_val=1500)
    on, orc, rv, rt, rs, comparable, _ = run_online(tp, wl, data, pk, X_test, "loss", m_ens=6, p_base=2,
                                                    p_ens=2, epochs=4)
    if comparable:
        check_best(on, orc, data, X_test, rv, rt, rs)


def test_online_stops_when_no_member_is_left(tp):
    """All learning rates 0 and p_base = 0: the second epoch repeats every
    score, removes every member and stops; further epochs are refused."""
    wl, data, pk, X_test = setup(tp, "tiny", "bf16", lr_zero=range(8))
    on, orc, rv, rt, rs, comparable, n = run_online(tp, wl, data, pk, X_test, "loss", m_ens=4, p_base=0,
                                                    p_ens=10, epochs=5)
    assert comparable and n == 2 and on.info()["stop"] == 1 and on.info()["n_active"] == 0
    with pytest.raises(tp.TabpackError):
        on.epoch(data["X_val"], data["y_val"])
    check_best(on, orc, data, X_test, rv, rt, rs)


def test_snapshot_restore_round_trip(tp):
    wl, data, pk, X_test = setup(tp, "tiny", "bf16")
    snap = pk.snapshot(2).clone()
    W0, b0 = pk.get_params(2, 0)
    p0 = pk.predict(X_test).cpu().numpy()
    for s, idx in enumerate(batch_indices(wl.n_train, wl.batch, 1)):
        pk.train_step(data["X_train"], torch.from_numpy(idx).cuda(), data["y_train"], s)
    assert not np.array_equal(pk.get_params(2, 0)[0], W0)
    pk.restore(2, snap)
    W1, b1 = pk.get_params(2, 0)
    assert np.array_equal(W1, W0) and np.array_equal(b1, b0)
    assert np.array_equal(pk.snapshot(2).cpu().numpy(), snap.cpu().numpy())
    assert np.array_equal(pk.predict(X_test).cpu().numpy()[2], p0[2])
    with pytest.raises(ValueError):
        pk.restore(2, snap[:-1])
