"""Pins of the oracle's online ensemble (Sec. 3.5 "Online ensemble", Sec. 3.6
early stopping) on hand-built validation predictions whose outcomes follow
from the paper's rules by hand: a regression target of zeros makes a
constant prediction c score c^2 (MSE), so every score below is known in
closed form."""
import math

import numpy as np
import pytest

from oracle.online import OnlineEnsemble


def preds_of(*rows):
    """[m, N, 1] float32 from per-member row lists."""
    return np.asarray(rows, dtype=np.float32)[:, :, None]


def test_previous_ensemble_joins_the_pool():
    """A model's epoch-1 and epoch-2 states are two candidates: with
    predictions a and -a they average to the target exactly."""
    y = np.zeros(2, dtype=np.float32)
    o = OnlineEnsemble(2, "regression", "loss", m_ens=4, p_base=10, p_ens=10)
    r1 = o.epoch_end(preds_of([0.5, -0.5], [2.0, 2.0]), y)
    assert r1["selected"] == [(0, 1)] and r1["score"] == 0.25
    assert r1["pool"] == [(0, 1), (1, 1)]
    r2 = o.epoch_end(preds_of([-0.5, 0.5], [2.0, 2.0]), y)
    # pool: (0,2) 0.25, (1,2) 4, (0,1) 0.25 -> tie to the lowest index, then (0,1) gives 0
    assert r2["pool"] == [(0, 2), (1, 2), (0, 1)]
    assert r2["selected"] == [(0, 2), (0, 1)] and r2["score"] == 0.0
    assert r2["improved"] and o.best == [(0, 2), (0, 1)] and o.best_epoch == 2
    r3 = o.epoch_end(preds_of([0.25, -0.25], [2.0, 2.0]), y)
    # three instances of model 0 average to (1/12, -1/12): worse than 0, the best stays
    assert r3["pool"] == [(0, 3), (1, 3), (0, 2), (0, 1)]
    assert r3["selected"] == [(0, 3), (0, 2), (0, 1)]
    assert r3["score"] == pytest.approx(1.0 / 144.0, rel=1e-6)
    assert not r3["improved"] and o.ens_bad == 1
    assert o.best == [(0, 2), (0, 1)] and o.best_score == 0.0 and o.best_epoch == 2


def test_base_model_patience():
    """Model 0 scores 1, .81, .9025, .9025, .81, ...: epochs 3, 4, 5 do not
    improve on .81 (equal is no improvement), so with p_base = 2 it leaves
    after epoch 5; model 1 keeps improving and stays."""
    y = np.zeros(1, dtype=np.float32)
    o = OnlineEnsemble(2, "regression", "loss", m_ens=1, p_base=2, p_ens=100)
    c0 = [1.0, 0.9, 0.95, 0.95, 0.9, np.nan]
    c1 = [0.5, 0.4, 0.3, 0.2, 0.1, 0.05]
    bad_after = [0, 0, 1, 2, 3]
    for k in range(5):
        r = o.epoch_end(preds_of([c0[k]], [c1[k]]), y)
        assert o.member_bad[0] == bad_after[k]
        assert r["removed"] == ([0] if k == 4 else [])
        assert o.active[0] == (k < 4)
        assert r["own"][0] == np.float32(c0[k]) * np.float32(c0[k])
    # epoch 6: model 0 is out of the pool; its (NaN) prediction is never read
    r = o.epoch_end(preds_of([c0[5]], [c1[5]]), y)
    assert r["pool"][0] == (1, 6) and all(m != 0 or e < 6 for m, e in r["pool"])
    assert math.isnan(r["own"][0]) and r["selected"] == [(1, 6)]
    assert o.active.tolist() == [False, True] and not r["stop"]


def test_base_model_patience_zero():
    """p_base = 0: the first epoch without improvement removes the model,
    and with no model left training stops."""
    y = np.zeros(1, dtype=np.float32)
    o = OnlineEnsemble(1, "regression", "loss", m_ens=2, p_base=0, p_ens=100)
    assert not o.epoch_end(preds_of([0.5]), y)["stop"]
    r = o.epoch_end(preds_of([0.5]), y)
    assert r["removed"] == [0] and r["stop"]
    with pytest.raises(RuntimeError):
        o.epoch_end(preds_of([0.1]), y)


def test_ensemble_patience_keeps_the_best():
    """One model that gets worse after epoch 1: the epoch-1 instance stays the
    ensemble (equal score, no improvement) and with p_ens = 1 training stops
    after the second epoch without improvement."""
    y = np.zeros(1, dtype=np.float32)
    o = OnlineEnsemble(1, "regression", "loss", m_ens=1, p_base=100, p_ens=1)
    r1 = o.epoch_end(preds_of([0.5]), y)
    assert r1["improved"] and not r1["stop"]
    r2 = o.epoch_end(preds_of([0.6]), y)
    assert r2["selected"] == [(0, 1)] and not r2["improved"] and o.ens_bad == 1 and not r2["stop"]
    r3 = o.epoch_end(preds_of([0.7]), y)
    assert r3["selected"] == [(0, 1)] and o.ens_bad == 2 and r3["stop"]
    assert o.best == [(0, 1)] and o.best_epoch == 1 and o.best_score == 0.25


def test_ensemble_improvement_resets_patience():
    y = np.zeros(1, dtype=np.float32)
    o = OnlineEnsemble(1, "regression", "loss", m_ens=1, p_base=100, p_ens=2)
    seq = [0.5, 0.6, 0.4, 0.45, 0.7, 0.8]
    bad = [0, 1, 0, 1, 2, 3]
    for k, c in enumerate(seq):
        r = o.epoch_end(preds_of([c]), y)
        assert o.ens_bad == bad[k]
        assert r["stop"] == (k == 5)
    assert o.best == [(0, 3)]


def test_accuracy_score_multiclass_pool():
    """Accuracy (a discrete score): the previous ensemble member is kept when
    the new states tie with it (ties go to the lowest candidate, and a tie is
    no improvement of the ensemble)."""
    y = np.array([0, 1, 2, 0], dtype=np.int32)
    eye = np.eye(3, dtype=np.float32)
    good = eye[y]                       # all four right
    o = OnlineEnsemble(2, "multiclass", "accuracy", m_ens=3, p_base=5, p_ens=5)
    r1 = o.epoch_end(np.stack([good, eye[[1, 1, 1, 1]]]), y)
    assert r1["selected"] == [(0, 1)] and r1["score"] == -1.0
    r2 = o.epoch_end(np.stack([good, good]), y)
    # three perfect candidates; the first is taken and no addition improves on -1
    assert r2["selected"] == [(0, 2)] and not r2["improved"] and o.best == [(0, 1)]
    # model 0 did not improve (equal), model 1 did
    assert o.member_bad.tolist() == [1, 0]


def test_auc_score_binary_pool():
    """ROC-AUC (score = -AUC): two models that each rank 3 of the 4
    positive-negative pairs right (AUC 3/4) but whose mean ranks all four
    right (AUC 1).  The first pick is the lower index among the tied
    singletons, the second model's addition strictly improves, and the base
    models' own scores are their single-model AUCs."""
    y = np.array([0, 0, 1, 1], dtype=np.int32)
    a = np.array([0.1, 0.5, 0.4, 0.9], dtype=np.float32)[:, None]   # 0.4 < 0.5: one pair wrong
    b = np.array([0.5, 0.1, 0.9, 0.4], dtype=np.float32)[:, None]   # 0.4 < 0.5: one pair wrong
    o = OnlineEnsemble(2, "binary", "auc", m_ens=4, p_base=3, p_ens=3)
    r = o.epoch_end(np.stack([a, b]), y)
    assert r["selected"] == [(0, 1), (1, 1)]
    assert r["score"] == -1.0 and r["improved"]
    assert o.member_best.tolist() == [-0.75, -0.75]
    # a model that ranks every pair right scores -1 alone and is picked first
    # (lowest pool index); nothing improves on -1, and a tie with the previous
    # ensemble's score is no improvement, so the best ensemble stays the first
    c = np.array([0.2, 0.3, 0.6, 0.7], dtype=np.float32)[:, None]
    r2 = o.epoch_end(np.stack([c, b]), y)
    assert r2["selected"][0] == (0, 2) and r2["score"] == -1.0 and not r2["improved"]
    assert o.best == [(0, 1), (1, 1)]
