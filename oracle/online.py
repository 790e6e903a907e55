"""Online ensemble with early stopping, restated on the CPU.

TEST INFRASTRUCTURE ONLY (as the rest of ``oracle/``): used by ``tests/``
to check the GPU library's online ensemble, never by the library.

What it follows:
  * Sec. 3.5 "Online ensemble": the ensemble is rebuilt from scratch once
    per epoch by greedy selection (Sec. 3.5 "Greedy ensembling") over a pool
    made of the latest states of the base models and the members of the
    previous epoch's ensemble; the same base model at different epochs gives
    different candidates.
  * Sec. 3.6 "Early stopping for the ensemble": training stops after
    p_ens + 1 consecutive epochs without an improvement of the ensemble's
    validation score.
  * Sec. 3.6 "Early stopping for the base models": a base model that has
    not improved its validation score for p_base + 1 consecutive epochs is
    removed from the pack.

Readings where the paper leaves a choice open:
  * a base model's validation score is the ensemble score of that model
    alone (the same score function the selection uses);
  * "improvement" is a strict decrease of the lower-is-better score against
    the best so far; NaN never improves;
  * removed base models leave the pool (their latest state would repeat
    a candidate already offered); their instances stay while they are
    ensemble members;
  * a member removed at an epoch still takes part in that epoch's pool;
  * the pool lists the active base models in index order and then the
    previous ensemble in its selection order (this fixes the tie-break:
    lowest candidate index);
  * the result of training is the best ensemble seen (lowest score,
    earliest on ties), together with its members' snapshots;
  * training also stops once no base model is left.

Scores come from ``oracle.greedy`` with fp32 per-row terms, the precision in
which the GPU scorer takes each decision; a base model's own score is the
greedy score of a one-candidate pool.
"""
from __future__ import annotations

import math

import numpy as np

from . import greedy


class OnlineEnsemble:
    def __init__(self, m, task, score, m_ens, p_base, p_ens, fp32_terms=True):
        self.m, self.task, self.score = int(m), task, score
        self.m_ens, self.p_base, self.p_ens = int(m_ens), int(p_base), int(p_ens)
        self.fp32_terms = fp32_terms
        self.active = np.ones(self.m, dtype=bool)
        self.member_best = np.full(self.m, np.inf)
        self.member_bad = np.zeros(self.m, dtype=np.int64)
        self.epoch = 0
        self.last = []                 # instances (member, epoch) of the last ensemble
        self.last_preds = None         # their predictions [n, N, d_out]
        self.best = []
        self.best_score = math.inf
        self.best_epoch = 0
        self.ens_bad = 0
        self.stop = False

    def _own_score(self, p, y):
        _, fin, _, _ = greedy(p[None], y, self.task, self.score, m_ens=1, fp32_terms=self.fp32_terms)
        return fin

    def epoch_end(self, live_preds, y):
        """live_preds: float32 [m, N, d_out], the base models' current
        validation predictions (rows of removed models are ignored)."""
        if self.stop:
            raise RuntimeError("training has stopped")
        live_preds = np.asarray(live_preds, dtype=np.float32)
        e = self.epoch + 1
        act = [i for i in range(self.m) if self.active[i]]
        if not act:
            raise RuntimeError("no active base model")
        # the pool: current states of the active models, then the last ensemble
        cands = [(i, e) for i in act] + list(self.last)
        parts = [live_preds[act]]
        if self.last:
            parts.append(self.last_preds)
        pool = np.concatenate(parts, axis=0)
        sel, fin, step_best, step_gap = greedy(pool, y, self.task, self.score, m_ens=self.m_ens,
                                               fp32_terms=self.fp32_terms)
        # base-model early stopping
        own = np.full(self.m, np.nan)
        removed = []
        for i in act:
            s = self._own_score(live_preds[i], y)
            own[i] = s
            if s < self.member_best[i]:
                self.member_best[i] = s
                self.member_bad[i] = 0
            else:
                self.member_bad[i] += 1
            if self.member_bad[i] >= self.p_base + 1:
                removed.append(i)
        # the rebuilt ensemble and ensemble early stopping
        now = [cands[c] for c in sel]
        improved = len(sel) > 0 and fin < self.best_score
        if improved:
            self.best, self.best_score, self.best_epoch, self.ens_bad = list(now), fin, e, 0
        else:
            self.ens_bad += 1
        self.last = now
        self.last_preds = pool[sel].copy()
        self.epoch = e
        for i in removed:
            self.active[i] = False
        self.stop = self.ens_bad >= self.p_ens + 1 or not self.active.any()
        return {"epoch": e, "pool": cands, "selected": now, "score": fin if len(sel) else math.nan,
                "step_best": step_best, "step_gap": step_gap, "own": own, "removed": removed,
                "improved": improved, "stop": self.stop}
