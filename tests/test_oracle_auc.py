"""Pins of the oracle's ROC-AUC ensemble score (the TabPack-dagger
experiments rank binary tasks by ROC-AUC): the rank-sum form against the
pairwise Mann-Whitney count, closed cases and a hand-worked example with
ties."""
import numpy as np
import pytest

import oracle


def pairwise_auc(s, y):
    s = np.asarray(s, dtype=np.float32)
    pos, neg = s[y == 1], s[y == 0]
    return ((pos[:, None] > neg[None, :]).sum() + 0.5 * (pos[:, None] == neg[None, :]).sum()) / (len(pos) * len(neg))


@pytest.mark.parametrize("seed", range(6))
def test_rank_sum_equals_pairwise_count(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(2, 60))
    s = np.round(rng.uniform(0, 1, n), 1 if seed % 2 else 3)   # coarse rounding makes ties
    y = rng.integers(0, 2, n).astype(np.int32)
    y[0], y[1] = 0, 1
    assert oracle.auc(s, y) == pytest.approx(pairwise_auc(s, y), abs=1e-15)


def test_closed_cases():
    y = np.array([0, 0, 0, 1, 1], dtype=np.int32)
    assert oracle.auc(np.array([0.1, 0.2, 0.3, 0.4, 0.5]), y) == 1.0
    assert oracle.auc(np.array([0.5, 0.4, 0.3, 0.2, 0.1]), y) == 0.0
    assert oracle.auc(np.full(5, 0.7), y) == 0.5
    assert np.isnan(oracle.auc(np.array([0.1, 0.2]), np.array([1, 1], dtype=np.int32)))


def test_hand_worked_with_ties():
    # positives 0.5, 0.9, 0.2 against negatives 0.5, 0.1:
    # (0.5: 1/2 + 1) + (0.9: 1 + 1) + (0.2: 0 + 1) = 4.5 of 6 pairs
    s = np.array([0.5, 0.5, 0.9, 0.1, 0.2])
    y = np.array([1, 0, 1, 0, 1], dtype=np.int32)
    assert oracle.auc(s, y) == 0.75


def test_monotone_transform_invariance():
    rng = np.random.default_rng(3)
    s = rng.uniform(-1, 1, 200)
    y = (rng.uniform(0, 1, 200) < 0.4).astype(np.int32)
    assert oracle.auc(s, y) == oracle.auc(s ** 3 + 2 * s, y)


@pytest.mark.parametrize("seed", range(4))
def test_matches_scikit_learn(seed):
    """Against scikit-learn's roc_auc_score (an independent implementation,
    trapezoidal area under the ROC curve, which counts ties as 1/2), on
    fp32 scores with and without ties."""
    metrics = pytest.importorskip("sklearn.metrics")
    rng = np.random.default_rng(100 + seed)
    n = int(rng.integers(5, 400))
    s = rng.uniform(0, 1, n).astype(np.float32)
    if seed % 2:
        s = (np.round(s * 16) / 16).astype(np.float32)
    y = rng.integers(0, 2, n).astype(np.int32)
    y[0], y[1] = 0, 1
    assert oracle.auc(s, y) == pytest.approx(metrics.roc_auc_score(y, s.astype(np.float64)), abs=1e-12)
