"""Pins for the oracle's greedy ensemble selection (Sec. 3.5).

Checked against an independent numpy scorer and brute-force search: the first
pick is the best singleton, every later pick is the best one-element
extension, the stopping rule is strict improvement, and on small pools the
greedy score is never better than the exhaustive optimum (equal on pools
built so that greedy is optimal).  Greedy is not optimal in general, so only
these provable relations are asserted.
"""
import itertools
import json
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def np_score(preds, subset, y, task, score):
    """Independent scorer: mean of the subset's predictions, then the metric."""
    ens = np.mean([preds[c].astype(np.float64) for c in subset], axis=0)
    if score == "auc":   # Mann-Whitney by pairs, on the fp32-rounded scores
        s32 = ens[:, 0].astype(np.float32)
        pos, neg = s32[y == 1], s32[y == 0]
        gt = (pos[:, None] > neg[None, :]).sum() + 0.5 * (pos[:, None] == neg[None, :]).sum()
        return -gt / (len(pos) * len(neg))
    if score == "accuracy":
        pred = np.argmax(ens, axis=1) if task == "multiclass" else (ens[:, 0] > 0.5).astype(int)
        return -np.mean(pred == y)
    if task == "regression":
        mse = np.mean((ens[:, 0] - y.astype(np.float64)) ** 2)
        return np.sqrt(mse) if score == "rmse" else mse
    q = ens[np.arange(len(y)), y] if task == "multiclass" else ens[:, 0]
    q = np.clip(q, 1e-7, 1 - 1e-7)
    if task == "multiclass":
        return -np.mean(np.log(q))
    return -np.mean(np.where(y == 1, np.log(q), np.log(1 - q)))


def make_pool(task, P, N, C, seed):
    rng = np.random.default_rng(seed)
    if task == "multiclass":
        logits = rng.standard_normal((P, N, C)) * 2
        preds = np.exp(logits) / np.exp(logits).sum(-1, keepdims=True)
        y = rng.integers(0, C, N)
    elif task == "binary":
        preds = 1 / (1 + np.exp(-2 * rng.standard_normal((P, N, 1))))
        y = rng.integers(0, 2, N)
    else:
        y = rng.standard_normal(N)
        preds = y[None, :, None] + rng.standard_normal((P, N, 1)) * rng.uniform(0.3, 1.5, (P, 1, 1))
    return preds.astype(np.float32), y.astype(np.float32 if task == "regression" else np.int32)


CASES = [("multiclass", "loss"), ("multiclass", "accuracy"), ("binary", "loss"),
         ("binary", "accuracy"), ("binary", "auc"), ("regression", "loss"), ("regression", "rmse")]


def test_worked_example(orc):
    g = json.load(open(os.path.join(GOLDEN, "greedy_worked_example.json")))
    preds = np.array(g["preds"], dtype=np.float32)
    y = np.array(g["y"], dtype=np.float32)
    for fp32_terms in (False, True):
        sel, fin, best, _ = orc.greedy(preds, y, g["task"], g["score"], g["m_ens"], fp32_terms)
        assert list(sel) == g["selected"]
        assert fin == g["final_score"]
        np.testing.assert_allclose(best, g["step_best"], rtol=1e-6, atol=1e-12)


@pytest.mark.parametrize("task,score", CASES)
@pytest.mark.parametrize("seed", range(4))
def test_each_step_is_best_extension(orc, task, score, seed):
    preds, y = make_pool(task, 9, 40, 4, seed)
    sel, fin, best, _ = orc.greedy(preds, y, task, score, m_ens=6)
    chosen = []
    cur = np.inf
    for k, c in enumerate(sel):
        cand = [j for j in range(len(preds)) if j not in chosen]
        scores = [np_score(preds, chosen + [j], y, task, score) for j in cand]
        j_best = cand[int(np.argmin(scores))]
        assert c == j_best
        assert abs(min(scores) - best[k]) < 1e-12
        if k > 0:
            assert min(scores) < cur
        chosen.append(c)
        cur = min(scores)
    # stopped for a reason: size limit or no strict improvement
    if len(sel) < 6:
        cand = [j for j in range(len(preds)) if j not in chosen]
        assert min(np_score(preds, chosen + [j], y, task, score) for j in cand) >= cur
    assert abs(fin - cur) < 1e-12


@pytest.mark.parametrize("task,score", CASES)
def test_single_pick_is_best_singleton(orc, task, score):
    preds, y = make_pool(task, 7, 33, 3, 11)
    sel, fin, _, _ = orc.greedy(preds, y, task, score, m_ens=1)
    singles = [np_score(preds, [c], y, task, score) for c in range(7)]
    assert list(sel) == [int(np.argmin(singles))]
    assert abs(fin - min(singles)) < 1e-12


@pytest.mark.parametrize("task,score", CASES)
@pytest.mark.parametrize("seed", range(3))
def test_never_beats_exhaustive_optimum(orc, task, score, seed):
    P = 6
    preds, y = make_pool(task, P, 25, 3, 100 + seed)
    sel, fin, _, _ = orc.greedy(preds, y, task, score, m_ens=P)
    best = min(np_score(preds, list(s), y, task, score)
               for r in range(1, P + 1) for s in itertools.combinations(range(P), r))
    assert fin >= best - 1e-12


def test_greedy_optimal_with_dominant_candidate(orc):
    """One perfect candidate plus duplicates and noisy ones: the optimum is
    the perfect candidate alone (any average with others is worse), and
    greedy finds it and stops."""
    rng = np.random.default_rng(0)
    N = 30
    y = rng.standard_normal(N).astype(np.float32)
    perfect = y[:, None].copy()
    pool = [y[:, None] + rng.standard_normal((N, 1)).astype(np.float32) for _ in range(3)]
    preds = np.stack([pool[0], pool[1], perfect, pool[2], pool[0].copy()]).astype(np.float32)
    sel, fin, _, _ = orc.greedy(preds, y, "regression", "loss", m_ens=5)
    assert list(sel) == [2] and fin == 0.0
    best = min(np_score(preds, list(s), y, "regression", "loss")
               for r in range(1, 6) for s in itertools.combinations(range(5), r))
    assert fin == best


def test_duplicates_tie_to_lowest_index(orc):
    preds, y = make_pool("multiclass", 4, 50, 3, 5)
    dup = np.concatenate([preds, preds], axis=0)        # candidates c and c + 4 identical
    sel, _, _, _ = orc.greedy(dup, y, "multiclass", "loss", m_ens=8)
    first = orc.greedy(preds, y, "multiclass", "loss", m_ens=1)[0][0]
    assert sel[0] == first
    # each duplicate pair is entered lower index first
    for c in sel:
        if c >= 4:
            assert (c - 4) in list(sel[:list(sel).index(c)])


@pytest.mark.parametrize("task,score", CASES)
@pytest.mark.parametrize("seed", range(3))
def test_fp32_terms_agree_with_plain_definition(orc, task, score, seed):
    preds, y = make_pool(task, 12, 300, 5, 40 + seed)
    a = orc.greedy(preds, y, task, score, m_ens=8, fp32_terms=False)
    b = orc.greedy(preds, y, task, score, m_ens=8, fp32_terms=True)
    # same decisions wherever the plain definition's margin is not a near-tie
    k = 0
    while k < min(len(a[0]), len(b[0])) and a[0][k] == b[0][k]:
        k += 1
    if k < max(len(a[0]), len(b[0])):
        assert a[3][k] < 1e-5 * max(1.0, abs(a[2][k]))
    assert abs(a[1] - b[1]) < 1e-5 * max(1.0, abs(a[1]))


def test_ensemble_score_matches_numpy(orc):
    for task, score in CASES:
        preds, y = make_pool(task, 5, 20, 4, 9)
        for subset in ([0], [1, 3], [4, 2, 0]):
            got = orc.ensemble_score(preds, subset, y, task, score)
            assert abs(got - np_score(preds, subset, y, task, score)) < 1e-12


def test_rejects_invalid(orc):
    preds, y = make_pool("regression", 3, 10, 1, 0)
    with pytest.raises(ValueError):
        orc.greedy(preds, y, "regression", "accuracy", 2)
    with pytest.raises(ValueError):
        orc.greedy(preds, y, "regression", "loss", 0)
