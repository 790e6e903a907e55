"""ctypes wrapper of the CPU fp64 oracle (``tabpack_oracle.c``).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py``.  The GPU library never imports,
links or calls anything in this package, and this package never touches the
GPU library.

The oracle restates the method of "TabPack: Efficient Hyperparameter
Ensembles for Tabular Deep Learning": the model pack (Sec. 3.3), the
optimizer pack (Sec. 3.4), per-member losses (Sec. 3.6) and greedy ensemble
selection (Sec. 3.5).  See ``tabpack_oracle.h`` for the exact readings.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "tabpack_oracle.c")
_HDR = os.path.join(_HERE, "tabpack_oracle.h")
LIB_PATH = os.path.join(_HERE, "liboracle.so")

BINARY, MULTICLASS, REGRESSION = 0, 1, 2
SCORE_LOSS, SCORE_ACCURACY, SCORE_RMSE, SCORE_AUC = 0, 1, 2, 3
TASKS = {"binary": BINARY, "multiclass": MULTICLASS, "regression": REGRESSION}
SCORES = {"loss": SCORE_LOSS, "accuracy": SCORE_ACCURACY, "rmse": SCORE_RMSE, "auc": SCORE_AUC}

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain C11, IEEE fp64: no fast-math and no
    FMA contraction, so x86-64 and aarch64 hosts give the same results)."""
    stale = (not os.path.exists(LIB_PATH)) or any(
        os.path.getmtime(p) > os.path.getmtime(LIB_PATH) for p in (_SRC, _HDR))
    if force or stale:
        tmp = LIB_PATH + f".{os.getpid()}.tmp"
        cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
               "-ffp-contract=off", "-fno-fast-math", "-Wall", "-Wno-unused-function",
               "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, LIB_PATH)
    return LIB_PATH


class _Config(ctypes.Structure):
    _fields_ = [("m", ctypes.c_int32), ("d_in", ctypes.c_int32), ("d_out", ctypes.c_int32),
                ("task", ctypes.c_int32), ("seed", ctypes.c_uint64),
                ("beta1", ctypes.c_double), ("beta2", ctypes.c_double), ("eps", ctypes.c_double),
                ("wd_on_bias", ctypes.c_int32), ("bf16_storage", ctypes.c_int32)]


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = ctypes.CDLL(LIB_PATH)
            P = ctypes.c_void_p
            i32, i64, u32, u64, f64 = (ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32,
                                       ctypes.c_uint64, ctypes.c_double)
            sig = {
                "orc_philox4x32_10": (None, [P, P, P]),
                "orc_dropout_keep": (ctypes.c_int, [u64, u32, u32, u32, u32, u32, ctypes.c_float]),
                "orc_round_bf16": (f64, [f64]),
                "orc_dropout_mask": (None, [u64, u32, u32, u32, i32, i32, ctypes.c_float, P]),
                "orc_create": (P, [ctypes.POINTER(_Config), P, P, P, P, P, P]),
                "orc_destroy": (None, [P]),
                "orc_init_value": (f64, [u64, u32, u32, u32, i32]),
                "orc_train_step": (ctypes.c_int, [P, P, i64, P, P, P, i32, u32, i32, P]),
                "orc_train_step_stacked": (ctypes.c_int, [P, P, i64, P, P, P, i32, u32, i32, P]),
                "orc_set_muon": (ctypes.c_int, [P, P, ctypes.c_double, i32]),
                "orc_auc": (ctypes.c_double, [P, P, i64]),
                "orc_create_emb": (P, [ctypes.POINTER(_Config), P, P, P, P, P, P, P, P]),
                "orc_get_emb": (ctypes.c_int, [P, i32, i32, P]),
                "orc_set_emb": (ctypes.c_int, [P, i32, P]),
                "orc_newton_schulz": (None, [P, i32, i32, i32, i32, P]),
                "orc_get_muon_dir": (ctypes.c_int, [P, i32, i32, P]),
                "orc_predict": (ctypes.c_int, [P, P, i64, P]),
                "orc_set_active": (ctypes.c_int, [P, P]),
                "orc_adamw_apply": (None, [P, P, P, P, i64, i64, f64, f64, f64, f64, f64]),
                "orc_get_params": (ctypes.c_int, [P, i32, i32, P, P]),
                "orc_set_params": (ctypes.c_int, [P, i32, i32, P, P]),
                "orc_get_grads": (ctypes.c_int, [P, i32, i32, P, P]),
                "orc_get_adam_state": (ctypes.c_int, [P, i32, i32, P, P, P, P]),
                "orc_get_logits": (ctypes.c_int, [P, i32, P]),
                "orc_get_keep": (ctypes.c_int, [P, i32, i32, P]),
                "orc_get_margin": (f64, [P, i32]),
                "orc_get_preact": (ctypes.c_int, [P, i32, i32, P]),
                "orc_member_steps": (i64, [P, i32]),
                "orc_greedy": (ctypes.c_int, [P, i32, i64, i32, P, P, i32, i32, i32, i32,
                                              P, P, P, P, P]),
                "orc_ensemble_score": (f64, [P, P, i32, i64, i32, P, P, i32, i32]),
            }
            for name, (res, args) in sig.items():
                fn = getattr(L, name)
                fn.restype = res
                fn.argtypes = args
            _lib = L
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def philox4x32_10(ctr, key):
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib().orc_philox4x32_10(_ptr(c), _ptr(k), _ptr(out))
    return out


def dropout_keep(seed, member_id, layer, step, row, col, p) -> int:
    return int(lib().orc_dropout_keep(seed, member_id, layer, step, row, col, float(p)))


def dropout_mask(seed, member_id, layer, step, B, w, p):
    """Keep mask [B, w] (uint8, 1 = keep) of one hidden layer at one step."""
    out = np.zeros((int(B), int(w)), dtype=np.uint8)
    lib().orc_dropout_mask(int(seed), int(member_id), int(layer), int(step), int(B), int(w), float(p), _ptr(out))
    return out


def round_bf16(x: float) -> float:
    return float(lib().orc_round_bf16(float(x)))


def init_value(seed, member_id, layer, e, fan_in) -> float:
    return float(lib().orc_init_value(seed, member_id, layer, e, fan_in))


def adamw_apply(p, g, t, lr, wd, m=None, v=None, beta1=0.9, beta2=0.999, eps=1e-8):
    """One AdamW step (Sec. 3.4; PyTorch semantics) of parameters p with
    gradients g at step count t, from moments m, v (zeros if None), in fp64.
    Returns the new (p, m, v)."""
    p = np.array(p, dtype=np.float64, copy=True).ravel()
    g = np.ascontiguousarray(g, dtype=np.float64).ravel()
    m = np.zeros_like(p) if m is None else np.array(m, dtype=np.float64, copy=True).ravel()
    v = np.zeros_like(p) if v is None else np.array(v, dtype=np.float64, copy=True).ravel()
    if not (p.size == g.size == m.size == v.size):
        raise ValueError("shape mismatch")
    lib().orc_adamw_apply(_ptr(p), _ptr(m), _ptr(v), _ptr(g), p.size, int(t), float(lr), float(wd),
                          float(beta1), float(beta2), float(eps))
    return p, m, v


def _labels(task, y):
    if task == REGRESSION:
        return None, np.ascontiguousarray(y, dtype=np.float32)
    return np.ascontiguousarray(y, dtype=np.int32), None


class OraclePack:
    """A pack of m base MLPs with per-member hyperparameters (CPU, fp64)."""

    def __init__(self, d_in, d_out, task, depth, width, dropout, lr, wd, seed,
                 beta1=0.9, beta2=0.999, eps=1e-8, wd_on_bias=True, bf16_storage=False,
                 member_id=None, d_emb=None, freq=None):
        """d_emb [m] and freq (the members' initial embedding frequencies,
        d_in x (d_emb[i] - 1) each, concatenated): periodic embeddings."""
        self.task = TASKS[task] if isinstance(task, str) else int(task)
        self.depth = np.ascontiguousarray(depth, dtype=np.int32)
        self.width = np.ascontiguousarray(width, dtype=np.int32)
        self.m = len(self.depth)
        self.d_in, self.d_out = int(d_in), int(d_out)
        cfg = _Config(self.m, self.d_in, self.d_out, self.task, int(seed), beta1, beta2, eps,
                      int(bool(wd_on_bias)), int(bool(bf16_storage)))
        drop = np.ascontiguousarray(dropout, dtype=np.float32)
        lr_ = np.ascontiguousarray(lr, dtype=np.float32)
        wd_ = np.ascontiguousarray(wd, dtype=np.float32)
        mid = None if member_id is None else np.ascontiguousarray(member_id, dtype=np.int32)
        self.d_emb = None
        if d_emb is None:
            h = lib().orc_create(ctypes.byref(cfg), _ptr(self.depth), _ptr(self.width), _ptr(drop),
                                 _ptr(lr_), _ptr(wd_), _ptr(mid))
        else:
            self.d_emb = np.ascontiguousarray(d_emb, dtype=np.int32)
            fr = np.ascontiguousarray(freq, dtype=np.float64).ravel()
            if fr.size != int(np.sum(self.d_in * (self.d_emb - 1))) or np.any(self.d_emb < 1):
                raise ValueError("freq must hold d_in x (d_emb - 1) values per member; d_emb >= 1")
            h = lib().orc_create_emb(ctypes.byref(cfg), _ptr(self.depth), _ptr(self.width), _ptr(drop),
                                     _ptr(lr_), _ptr(wd_), _ptr(mid), _ptr(self.d_emb), _ptr(fr))
        if not h:
            raise ValueError("oracle rejected the pack configuration")
        self._h = ctypes.c_void_p(h)
        self._B = 0

    def __del__(self):
        h = getattr(self, "_h", None)
        if h is not None and _lib is not None:
            _lib.orc_destroy(h)
            self._h = None

    def layer_shape(self, member, layer):
        L, w = int(self.depth[member]), int(self.width[member])
        n_in = (self.d_in * (int(self.d_emb[member]) if self.d_emb is not None else 1)) if layer == 0 else w
        n_out = self.d_out if layer == L else w
        return n_out, n_in

    def train_step(self, X, idx, y, step, update=True):
        """idx [B] (one batch for every member) or [m, B] (member i's batch in
        row i, Sec. 3.6 stacked base batches)."""
        X = np.ascontiguousarray(X, dtype=np.float32)
        idx = np.ascontiguousarray(idx, dtype=np.int32)
        yi, yf = _labels(self.task, y)
        loss = np.zeros(self.m, dtype=np.float64)
        if idx.ndim == 2:
            if idx.shape[0] != self.m:
                raise ValueError("stacked idx must have one row per member")
            fn, B = lib().orc_train_step_stacked, idx.shape[1]
        else:
            fn, B = lib().orc_train_step, len(idx)
        rc = fn(self._h, _ptr(X), X.shape[0], _ptr(idx), _ptr(yi), _ptr(yf), B, int(step), int(bool(update)),
                _ptr(loss))
        if rc:
            raise ValueError("oracle train_step rejected its arguments")
        self._B = B
        return loss

    def predict(self, X):
        X = np.ascontiguousarray(X, dtype=np.float32)
        out = np.zeros((self.m, X.shape[0], self.d_out), dtype=np.float64)
        if lib().orc_predict(self._h, _ptr(X), X.shape[0], _ptr(out)):
            raise ValueError("oracle predict rejected its arguments")
        return out

    def set_active(self, active):
        a = np.ascontiguousarray(active, dtype=np.uint8)
        lib().orc_set_active(self._h, _ptr(a))

    def emb(self, member, grads=False):
        """(w, b, alpha, beta) of a member's embeddings (or their gradients)."""
        d, n = int(self.d_emb[member]), self.d_in
        out = np.zeros(n * (4 * d - 2), dtype=np.float64)
        if lib().orc_get_emb(self._h, int(member), int(bool(grads)), _ptr(out)):
            raise ValueError("no embeddings")
        k = n * (d - 1)
        return (out[:k].reshape(n, d - 1), out[k:2 * k].reshape(n, d - 1), out[2 * k:2 * k + n * d].reshape(n, d),
                out[2 * k + n * d:].reshape(n, d))

    def set_emb(self, member, w, b, alpha, beta):
        flat = np.concatenate([np.ravel(w), np.ravel(b), np.ravel(alpha), np.ravel(beta)]).astype(np.float64)
        if lib().orc_set_emb(self._h, int(member), _ptr(flat)):
            raise ValueError("no embeddings")

    def set_muon(self, lr_muon, momentum=0.95, ns_steps=5):
        """Muon for the hidden-layer weights from now on (Sec. 3.4)."""
        lr = np.ascontiguousarray(lr_muon, dtype=np.float64)
        if lib().orc_set_muon(self._h, _ptr(lr), float(momentum), int(ns_steps)):
            raise ValueError("oracle set_muon rejected its arguments")

    def muon_dir(self, member, layer):
        n_out, n_in = self.layer_shape(member, layer)
        out = np.zeros((n_out, n_in), dtype=np.float64)
        if lib().orc_get_muon_dir(self._h, int(member), int(layer), _ptr(out)):
            raise ValueError("no Muon direction for this layer")
        return out

    def _two(self, fn, member, layer):
        n_out, n_in = self.layer_shape(member, layer)
        W = np.zeros((n_out, n_in), dtype=np.float64)
        b = np.zeros(n_out, dtype=np.float64)
        if fn(self._h, member, layer, _ptr(W), _ptr(b)):
            raise IndexError((member, layer))
        return W, b

    def get_params(self, member, layer):
        return self._two(lib().orc_get_params, member, layer)

    def get_grads(self, member, layer):
        return self._two(lib().orc_get_grads, member, layer)

    def set_params(self, member, layer, W, b):
        W = np.ascontiguousarray(W, dtype=np.float64)
        b = np.ascontiguousarray(b, dtype=np.float64)
        if W.shape != self.layer_shape(member, layer) or b.shape != (W.shape[0],):
            raise ValueError("shape mismatch")
        if lib().orc_set_params(self._h, member, layer, _ptr(W), _ptr(b)):
            raise IndexError((member, layer))

    def get_adam_state(self, member, layer):
        n_out, n_in = self.layer_shape(member, layer)
        mW = np.zeros((n_out, n_in)); vW = np.zeros((n_out, n_in))
        mb = np.zeros(n_out); vb = np.zeros(n_out)
        lib().orc_get_adam_state(self._h, member, layer, _ptr(mW), _ptr(vW), _ptr(mb), _ptr(vb))
        return mW, vW, mb, vb

    def logits(self, member):
        out = np.zeros((self._B, self.d_out), dtype=np.float64)
        if lib().orc_get_logits(self._h, member, _ptr(out)):
            raise IndexError(member)
        return out

    def keep(self, member, layer):
        out = np.zeros((self._B, int(self.width[member])), dtype=np.uint8)
        if lib().orc_get_keep(self._h, member, layer, _ptr(out)):
            raise IndexError((member, layer))
        return out

    def preact(self, member, layer):
        out = np.zeros((self._B, int(self.width[member])), dtype=np.float64)
        if lib().orc_get_preact(self._h, member, layer, _ptr(out)):
            raise IndexError((member, layer))
        return out

    def margin(self, member):
        return float(lib().orc_get_margin(self._h, member))

    def member_steps(self, member):
        return int(lib().orc_member_steps(self._h, member))


def auc(e, y):
    """ROC-AUC of scores e for 0/1 labels y (ranked in fp32, midranks for ties)."""
    e = np.ascontiguousarray(e, dtype=np.float64)
    y = np.ascontiguousarray(y, dtype=np.int32)
    return float(lib().orc_auc(_ptr(e), _ptr(y), len(e)))


def newton_schulz(U, steps=5, bf16=False):
    """Muon's orthogonalized direction of U (oracle; see tabpack_oracle.c)."""
    U = np.ascontiguousarray(U, dtype=np.float64)
    O = np.zeros_like(U)
    lib().orc_newton_schulz(_ptr(U), U.shape[0], U.shape[1], int(steps), int(bool(bf16)), _ptr(O))
    return O


def greedy(preds, y, task, score="loss", m_ens=32, fp32_terms=False):
    """Greedy ensemble selection (Sec. 3.5).  Returns (selected, final_score,
    step_best, step_gap)."""
    preds = np.ascontiguousarray(preds, dtype=np.float32)
    P, N, d_out = preds.shape
    t = TASKS[task] if isinstance(task, str) else int(task)
    s = SCORES[score] if isinstance(score, str) else int(score)
    yi, yf = _labels(t, y)
    sel = np.zeros(m_ens, dtype=np.int32)
    n = ctypes.c_int32(0)
    fin = ctypes.c_double(0.0)
    best = np.full(m_ens, np.nan)
    gap = np.full(m_ens, np.nan)
    rc = lib().orc_greedy(_ptr(preds), P, N, d_out, _ptr(yi), _ptr(yf), t, s, m_ens,
                          int(bool(fp32_terms)), _ptr(sel), ctypes.byref(n), ctypes.byref(fin),
                          _ptr(best), _ptr(gap))
    if rc:
        raise ValueError("oracle greedy rejected its arguments")
    k = n.value
    return sel[:k].copy(), fin.value, best[:k].copy(), gap[:k].copy()


def ensemble_score(preds, subset, y, task, score="loss"):
    preds = np.ascontiguousarray(preds, dtype=np.float32)
    P, N, d_out = preds.shape
    t = TASKS[task] if isinstance(task, str) else int(task)
    s = SCORES[score] if isinstance(score, str) else int(score)
    yi, yf = _labels(t, y)
    sub = np.ascontiguousarray(subset, dtype=np.int32)
    return float(lib().orc_ensemble_score(_ptr(preds), _ptr(sub), len(sub), N, d_out,
                                          _ptr(yi), _ptr(yf), t, s))
