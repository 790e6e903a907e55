"""Comparison rules of the GPU parity tests (imported by the test modules).

Floats.  The relative error of an entry is |g - o| / max(|o|, rms(o)) (the
tensor's rms floors entries near zero: a computed entry's rounding error
scales with the terms summed into it, not with the entry itself).

fp32 mode is held to the fp64 oracle at 1e-4.

bf16 mode is held to the fp64 oracle run in exact arithmetic (the paper's
method with no rounding), at 2e-2 per entry.  Storing activations, weights
and gradients in bf16 (8 significant bits) can itself move a result further
than that from the exact one, and the oracle shows by how much without the
GPU: its bf16-storage mode rounds the same stored values (the paper's method
with bf16 storage) and is compared with its exact mode.  A GPU tensor may
exceed 2e-2 only where that oracle-only distance does too, and then it may
be at most twice as far from the exact result as the oracle's own bf16 model
is, entrywise and norm-wise.  The comparison with the bf16-storage oracle
(same storage points) is kept as a second, diagnostic assertion at 2e-2.

ReLU decisions at a near-tie.  A pre-activation within rounding of zero may
be kept on one side and cut on the other; both are valid subgradients.  The
tests read the GPU's stored activations, find every decision that differs
from the oracle's, and require each to sit at an oracle near-tie.  The
bound comes from the oracle alone: 1e-5 rms(Z) in fp32 mode (fp32 rounding
of sums of a few hundred terms stays below 1e-6 rms), and in bf16 mode twice
the largest distance between the pre-activations of the oracle's
bf16-storage and exact modes in that layer.  A flip at (row b, unit j) of
layer l changes row j of layer l's weight gradient by one of B batch terms;
in bf16 mode those rows are held to the bar norm-wise and every other entry
entrywise; in fp32 mode a member with a flip is held norm-wise per tensor.
"""
from __future__ import annotations

import numpy as np

import oracle

TOL = {"fp32": 1e-4, "bf16": 2e-2}
TIE_FP32 = 1e-5

# per tensor kind: the largest GPU-vs-exact error and the oracle's own
# bf16-vs-exact error of the same tensor (bf16 mode), for the test report
STATS: dict = {}


def rms(a) -> float:
    a = np.asarray(a, dtype=np.float64)
    return float(np.sqrt(np.mean(a ** 2))) if a.size else 0.0


def rel_err(got, ref, rows=None) -> float:
    """Largest floored relative error; rows (bool [n_rows]) selects rows of
    a 2-D tensor to compare (the floor stays the whole tensor's rms)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    if ref.size == 0:
        return 0.0
    r = rms(ref)
    floor = np.maximum(np.abs(ref), r if r > 0 else 1e-30)
    e = np.abs(got - ref) / floor
    if rows is not None:
        e = e[rows]
    return float(np.max(e)) if e.size else 0.0


def nrm_err(got, ref) -> float:
    got = np.asarray(got, dtype=np.float64).ravel()
    ref = np.asarray(ref, dtype=np.float64).ravel()
    return float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30))


class Oracles:
    """The exact fp64 oracle of a pack (`ex`) and, in bf16 mode, the oracle's
    bf16-storage model of the same pack (`bst`), stepped together.  Every
    other attribute reads the exact oracle."""

    def __init__(self, prec, *args, **kw):
        kw.pop("bf16_storage", None)
        self.prec = prec
        self.ex = oracle.OraclePack(*args, bf16_storage=False, **kw)
        self.bst = oracle.OraclePack(*args, bf16_storage=True, **kw) if prec == "bf16" else None
        self.loss_bst = None
        self.last_loss = None

    def __getattr__(self, name):
        return getattr(self.ex, name)

    def _both(self, name, *a, **k):
        r = getattr(self.ex, name)(*a, **k)
        if self.bst is not None:
            getattr(self.bst, name)(*a, **k)
        return r

    def train_step(self, *a, **k):
        loss = self.ex.train_step(*a, **k)
        self.last_loss = loss
        if self.bst is not None:
            self.loss_bst = self.bst.train_step(*a, **k)
        return loss

    def set_active(self, active):
        return self._both("set_active", active)

    def set_params(self, *a):
        return self._both("set_params", *a)

    def set_emb(self, *a):
        return self._both("set_emb", *a)

    def set_muon(self, *a, **k):
        return self._both("set_muon", *a, **k)

    def tie_bound(self, oi, l) -> float:
        """Oracle-only near-tie half-width of layer l's pre-activations, in
        units of their rms: 1e-5 (fp32 mode) or twice the largest
        |Z_bf16storage - Z_exact| / rms(Z_exact) (bf16 mode)."""
        if self.bst is None:
            return TIE_FP32
        zx = self.ex.preact(oi, l)
        zb = self.bst.preact(oi, l)
        r = rms(zx)
        return 2.0 * float(np.max(np.abs(zb - zx))) / r if r > 0 else 0.0


def flip_sites(pk, i, orc_side, oi, l, bound):
    """Decisions of GPU member i, layer l, that differ from oracle member
    oi's (bool [B, w]); asserts each lies within bound * rms(Z) of zero."""
    Hg = pk.debug_activations(i, l).astype(np.float64)
    Zo = orc_side.preact(oi, l)
    keep = orc_side.keep(oi, l) > 0
    diff = (Hg > 0) != ((Zo > 0) & keep)
    if diff.any():
        zr = rms(Zo)
        worst = float(np.max(np.abs(Zo[diff])) / zr)
        assert worst <= bound, ("decision flipped away from an oracle near-tie", i, l, worst, bound)
    return diff


def _record(kind, e_g, e_r):
    s = STATS.setdefault(kind, [0.0, 0.0])
    s[0] = max(s[0], e_g)
    s[1] = max(s[1], e_r)


def check_bf16_vs_exact(kind, g, ob, ox, problems, key):
    """Primary bf16 bar: GPU g against the exact oracle ox, at 2e-2 or, where
    the oracle's own bf16-storage result ob is further than that from ox,
    within twice ob's distance (entrywise and norm-wise)."""
    tol = TOL["bf16"]
    e_g, e_r = rel_err(g, ox), rel_err(ob, ox)
    n_g, n_r = nrm_err(g, ox), nrm_err(ob, ox)
    _record(kind, e_g, e_r)
    if e_g > max(tol, 2.0 * e_r) or n_g > max(tol, 2.0 * n_r):
        problems.append((key, "vs exact", e_g, e_r, n_g, n_r))


def _check_flipped(g, o, flip_rows, tol, problems, key):
    """Entrywise outside the rows a flip touched, norm-wise over the tensor."""
    keep_rows = ~flip_rows
    e = rel_err(g, o, rows=keep_rows)
    n = nrm_err(g, o)
    if e > tol or n > tol:
        problems.append((key, int(flip_rows.sum()), e, n))


def compare_step(pk, orc: Oracles, hp, prec, loss_gpu, members=None, emb_grads=None):
    """One step's losses, logits and every gradient of GPU members `members`
    (default all) against oracle members 0, 1, ... (the oracle may hold only
    the sampled members; members are independent).  emb_grads(i, oi) ->
    list of (gpu, exact, bf16 storage) embedding gradient arrays, or None.
    Returns {member: [problems]}."""
    tol = TOL[prec]
    members = list(range(len(hp["depth"]))) if members is None else list(members)
    problems = {}
    for oi, i in enumerate(members):
        L = int(hp["depth"][i])
        p = []
        bounds = [orc.tie_bound(oi, l) for l in range(L)]
        # decisions flipped against the exact oracle (primary) and against
        # the bf16-storage oracle (diagnostic)
        flips_x = [flip_sites(pk, i, orc.ex, oi, l, bounds[l]) for l in range(L)]
        flips_b = [flip_sites(pk, i, orc.bst, oi, l, bounds[l]) for l in range(L)] if orc.bst is not None else None
        lg = float(loss_gpu[i])
        logit_g = pk.logits(i)
        grads_g = [pk.get_grads(i, l) for l in range(L + 1)]
        grads_x = [orc.ex.get_grads(oi, l) for l in range(L + 1)]
        if prec == "fp32":
            if abs(lg - orc.last_loss[oi]) / max(1.0, abs(orc.last_loss[oi])) > tol:
                p.append(("loss", lg, orc.last_loss[oi]))
            e = rel_err(logit_g, orc.ex.logits(oi))
            if e > tol:
                p.append(("logits", e))
            any_flip = any(f.any() for f in flips_x)
            for l in range(L + 1):
                (gW, gb), (oW, ob) = grads_g[l], grads_x[l]
                if not any_flip:
                    e = max(rel_err(gW, oW), rel_err(gb, ob))
                else:
                    e = nrm_err(np.concatenate([gW.ravel(), gb]), np.concatenate([oW.ravel(), ob]))
                if e > tol:
                    p.append(("grad", l, any_flip, e))
            if emb_grads is not None:
                for k, (g, ox, _) in enumerate(emb_grads(i, oi)):
                    e = nrm_err(g, ox) if any_flip else rel_err(g, ox)
                    if e > tol:
                        p.append(("emb grad", k, any_flip, e))
        else:
            lb = orc.loss_bst[oi]
            lxv = orc.last_loss[oi]
            # a member's mean loss: error relative to max(1, |loss|)
            e_g, e_r = abs(lg - lxv) / max(1.0, abs(lxv)), abs(lb - lxv) / max(1.0, abs(lxv))
            _record("loss", e_g, e_r)
            if e_g > max(tol, 2.0 * e_r):
                p.append(("loss", "vs exact", lg, lxv, lb))
            check_bf16_vs_exact("logits", logit_g, orc.bst.logits(oi), orc.ex.logits(oi), p, "logits")
            grads_b = [orc.bst.get_grads(oi, l) for l in range(L + 1)]
            flip_any = [f.any() for f in flips_b]
            for l in range(L + 1):
                kind = "grad hidden" if l < L else "grad head"
                # diagnostic: rows of layer l whose unit flipped against the
                # bf16 model are held to the bar norm-wise, and so is the
                # whole tensor when a layer above it flipped (the flip
                # changes one row of the back-propagated gradient below it)
                flip_rows = flips_b[l].any(axis=0) if l < L else np.zeros(grads_g[l][1].shape[0], dtype=bool)
                if any(flip_any[l + 1:]):
                    flip_rows = np.ones_like(flip_rows)
                for t, name in ((0, "W"), (1, "b")):
                    g, ox, ob = grads_g[l][t], grads_x[l][t], grads_b[l][t]
                    check_bf16_vs_exact(kind, g, ob, ox, p, ("grad", l, name))
                    _check_flipped(g, ob, flip_rows, tol, p, ("grad vs bf16 model", l, name))
            if abs(lg - lb) / max(1.0, abs(lb)) > tol:
                p.append(("loss vs bf16 model", lg, lb))
            e = rel_err(logit_g, orc.bst.logits(oi))
            if e > tol:
                p.append(("logits vs bf16 model", e))
            if emb_grads is not None:
                # a flipped decision changes one of B rows of dE, which every
                # embedding gradient sums: norm-wise then
                flip_b = any(flip_any)
                for k, (g, ox, ob) in enumerate(emb_grads(i, oi)):
                    check_bf16_vs_exact("emb grad", g, ob, ox, p, ("emb grad", k))
                    e = nrm_err(g, ob) if flip_b else rel_err(g, ob)
                    if e > tol:
                        p.append(("emb grad vs bf16 model", k, flip_b, e))
        if p:
            problems[i] = p
    return problems


def compare_params(pk, orc: Oracles, hp, prec, members=None, margin=None, oracle_index=None, extra=None,
                   diag_ratio=None):
    """Parameters after several steps: fp32 at 1e-4 against the exact oracle
    (a member whose oracle pre-activations came within 1e-5 rms of zero in
    some step -- margin[i] < 1e-5 -- may have taken the other subgradient
    there, and may be held at the bf16 bar; such members are returned; the
    oracle holds member members[k] at oracle_index[k], default k); bf16
    by check_bf16_vs_exact plus the bf16-storage oracle at 2e-2.  extra(i,
    oi) -> list of further (name, gpu, exact, bf16 storage) tensors of a
    member.  diag_ratio: a tensor that misses the 2e-2 diagnostic bar passes
    it when its norm-wise distance from the bf16-storage oracle is within
    diag_ratio times that oracle's own distance from the exact one (for
    parameters that start at zero, whose first Adam steps are +-lr by the
    sign of a gradient that may sit within rounding of zero).  Returns
    (largest error per member, problems, members held at the bf16 bar)."""
    tol = TOL[prec]
    members = list(range(len(hp["depth"]))) if members is None else list(members)
    oracle_index = list(range(len(members))) if oracle_index is None else list(oracle_index)
    errs, problems, relaxed = {}, {}, set()
    for oi, i in zip(oracle_index, members):
        p = []
        e_max = 0.0
        trip = []
        for l in range(int(hp["depth"][i]) + 1):
            gp, xp = pk.get_params(i, l), orc.ex.get_params(oi, l)
            bp = orc.bst.get_params(oi, l) if prec == "bf16" else (None, None)
            trip += [((l, "W"), gp[0], xp[0], bp[0]), ((l, "b"), gp[1], xp[1], bp[1])]
        if extra is not None:
            trip += [((name, ""), g, x, b) for name, g, x, b in extra(i, oi)]
        for (l, name), g, ox, ob in trip:
            if prec == "fp32":
                e = rel_err(g, ox)
                e_max = max(e_max, e)
                near_tie = margin is not None and margin[oi] < TIE_FP32
                if e > tol and near_tie and e <= TOL["bf16"]:
                    relaxed.add(i)
                elif e > tol:
                    p.append(("params", l, name, e))
            else:
                check_bf16_vs_exact("params", g, ob, ox, p, ("params", l, name))
                e = rel_err(g, ob)
                if e > tol and diag_ratio is not None and \
                        nrm_err(g, ob) <= max(diag_ratio * nrm_err(ob, ox), 1e-3):
                    e = 0.0
                e_max = max(e_max, e)
                if e > tol:
                    p.append(("params vs bf16 model", l, name, e))
        errs[i] = e_max
        if p:
            problems[i] = p
    return errs, problems, relaxed
