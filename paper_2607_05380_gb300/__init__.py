"""Python binding of the tabpack C ABI (``include/tabpack.h``).

Argument marshalling only: every step of the training path runs in the CUDA
kernels of ``libtabpack.so``; PyTorch provides device memory and streams.
The library must have been built (``build.build()``); importing the binding
without it raises, there is no fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

from . import build as _build

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = _build.LIB

TP_OK, TP_EINVAL, TP_ENOMEM, TP_ECUDA, TP_ESTATE, TP_ETIMEOUT, TP_ENOTSUP = range(7)
BINARY, MULTICLASS, REGRESSION = 0, 1, 2
BF16, FP32 = 0, 1
SCORE_LOSS, SCORE_ACCURACY, SCORE_RMSE, SCORE_AUC = 0, 1, 2, 3
TASKS = {"binary": BINARY, "multiclass": MULTICLASS, "regression": REGRESSION}
PRECISIONS = {"bf16": BF16, "fp32": FP32}
SCORES = {"loss": SCORE_LOSS, "accuracy": SCORE_ACCURACY, "rmse": SCORE_RMSE, "auc": SCORE_AUC}
PHASES = ["gather", "fwd", "head", "bwd", "bias", "adamw", "predict", "muon"]

# every entry point declared in include/tabpack.h
SYMBOLS = ["pack_create", "pack_destroy", "pack_set_stream", "pack_train_step", "pack_forward_backward",
           "pack_predict", "pack_select_greedy", "pack_select_greedy_static", "pack_set_active", "pack_get_params", "pack_set_params",
           "pack_get_grads", "pack_get_logits", "pack_debug_masks", "pack_debug_activations", "pack_profile_enable",
           "pack_profile_read", "pack_launch_count", "pack_sizes", "pack_last_error", "pack_member_size",
           "pack_snapshot", "pack_restore", "pack_get_config", "pack_member_hparams", "pack_get_active",
           "pack_get_stream", "pack_online_create", "pack_online_destroy", "pack_online_epoch", "pack_online_info",
           "pack_online_members", "pack_online_ensemble", "pack_online_snapshot", "pack_online_predict",
           "pack_online_last_error", "pack_train_step_stacked", "pack_forward_backward_stacked", "pack_set_muon",
           "pack_debug_muon_dir", "pack_create_emb", "pack_get_emb", "pack_set_emb", "pack_member_emb",
           "pack_debug_mask_arena", "pack_debug_philox", "pack_debug_gemm_timeout", "pack_debug_bias_path"]


class TabpackError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"tabpack status {status}: {msg}")
        self.status = status


class Config(ctypes.Structure):
    _fields_ = [("m", ctypes.c_int32), ("d_in", ctypes.c_int32), ("d_out", ctypes.c_int32),
                ("max_batch", ctypes.c_int32), ("task", ctypes.c_int32), ("precision", ctypes.c_int32),
                ("seed", ctypes.c_uint64), ("beta1", ctypes.c_float), ("beta2", ctypes.c_float),
                ("eps", ctypes.c_float), ("wd_on_bias", ctypes.c_int32), ("fuse_optimizer", ctypes.c_int32)]


class OnlineInfo(ctypes.Structure):
    _fields_ = [("epoch", ctypes.c_int32), ("stop", ctypes.c_int32), ("n_active", ctypes.c_int32),
                ("ens_bad", ctypes.c_int32), ("best_epoch", ctypes.c_int32), ("n_best", ctypes.c_int32),
                ("n_last", ctypes.c_int32), ("n_pool", ctypes.c_int32), ("best_score", ctypes.c_double),
                ("last_score", ctypes.c_double)]


_lib = None


def load_library(path: str = LIB_PATH):
    """Load libtabpack.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"libtabpack.so not built at {path}: run paper_2607_05380_gb300.build.build()")
    L = ctypes.CDLL(path)
    P, i32, i64, u32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32
    st = ctypes.c_int
    sig = {
        "pack_create": (st, [ctypes.POINTER(Config), P, P, P, P, P, P, ctypes.POINTER(P)]),
        "pack_destroy": (None, [P]),
        "pack_set_stream": (st, [P, P]),
        "pack_train_step": (st, [P, P, i64, P, P, i32, u32, P]),
        "pack_forward_backward": (st, [P, P, i64, P, P, i32, u32, P]),
        "pack_predict": (st, [P, P, i64, P]),
        "pack_select_greedy": (st, [P, i32, i64, i32, P, i32, i32, i32, P, P, P, P]),
        "pack_select_greedy_static": (st, [P, i32, i64, i32, P, i32, i32, i32, P, P, P, P]),
        "pack_set_active": (st, [P, P]),
        "pack_get_params": (st, [P, i32, i32, P, P]),
        "pack_set_params": (st, [P, i32, i32, P, P]),
        "pack_get_grads": (st, [P, i32, i32, P, P]),
        "pack_get_logits": (st, [P, i32, P]),
        "pack_debug_masks": (st, [P, i32, i32, u32, i32, P]),
        "pack_debug_activations": (st, [P, i32, i32, P]),
        "pack_profile_enable": (st, [P, i32]),
        "pack_profile_read": (st, [P, P, P, i32]),
        "pack_launch_count": (i64, [P]),
        "pack_sizes": (st, [P, P, P]),
        "pack_last_error": (ctypes.c_char_p, [P]),
        "pack_member_size": (st, [P, i32, P]),
        "pack_snapshot": (st, [P, i32, P]),
        "pack_restore": (st, [P, i32, P]),
        "pack_get_config": (st, [P, ctypes.POINTER(Config)]),
        "pack_member_hparams": (st, [P, i32, P, P, P, P, P]),
        "pack_get_active": (st, [P, P]),
        "pack_get_stream": (P, [P]),
        "pack_online_create": (st, [P, i64, i32, i32, i32, i32, ctypes.POINTER(P)]),
        "pack_online_destroy": (None, [P]),
        "pack_online_epoch": (st, [P, P, P, P]),
        "pack_online_info": (st, [P, ctypes.POINTER(OnlineInfo)]),
        "pack_online_members": (st, [P, P, P, P]),
        "pack_online_ensemble": (st, [P, i32, P, P, P, P]),
        "pack_online_snapshot": (st, [P, i32, P]),
        "pack_online_predict": (st, [P, P, i64, P]),
        "pack_online_last_error": (ctypes.c_char_p, [P]),
        "pack_train_step_stacked": (st, [P, P, i64, P, P, i32, u32, P]),
        "pack_set_muon": (st, [P, P, ctypes.c_float, i32]),
        "pack_debug_muon_dir": (st, [P, i32, i32, P]),
        "pack_forward_backward_stacked": (st, [P, P, i64, P, P, i32, u32, P]),
        "pack_create_emb": (st, [ctypes.POINTER(Config), P, P, P, P, P, P, P, P, ctypes.POINTER(P)]),
        "pack_get_emb": (st, [P, i32, i32, P]),
        "pack_set_emb": (st, [P, i32, P]),
        "pack_member_emb": (st, [P, i32, P]),
        "pack_debug_mask_arena": (st, [P, i32, i32, i32, P, P]),
        "pack_debug_philox": (st, [P, P, i32, P]),
        "pack_debug_gemm_timeout": (st, [P, ctypes.c_double, i32]),
        "pack_debug_bias_path": (st, [P, i32]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    _lib = L
    return L


def _check(status, handle=None):
    if status != TP_OK:
        msg = load_library().pack_last_error(handle)
        raise TabpackError(status, msg.decode() if msg else "")


def _dptr(t, dtype=None):
    """Device pointer of a contiguous CUDA tensor (None for None)."""
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"expected {dtype}, got {t.dtype}")
    return ctypes.c_void_p(t.data_ptr())


def _hptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _stream_ptr(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


class Pack:
    """A pack of m base MLPs with per-member hyperparameters on one GPU."""

    def __init__(self, d_in, d_out, task, depth, width, dropout, lr, wd, max_batch, seed=2,
                 precision="bf16", beta1=0.9, beta2=0.999, eps=1e-8, wd_on_bias=True, stream=None,
                 fuse_optimizer=False, d_emb=None, freq=None):
        """d_emb: per-member periodic embedding sizes (None: the members read
        the raw features); freq: their initial frequencies w, member after
        member [d_in, d_emb[i] - 1] (App. "Feature Embeddings")."""
        import torch
        L = load_library()
        self.torch = torch
        self.depth = np.ascontiguousarray(depth, dtype=np.int32)
        self.width = np.ascontiguousarray(width, dtype=np.int32)
        self.m = len(self.depth)
        self.d_in, self.d_out = int(d_in), int(d_out)
        self.task = TASKS[task] if isinstance(task, str) else int(task)
        self.precision = PRECISIONS[precision] if isinstance(precision, str) else int(precision)
        cfg = Config(self.m, self.d_in, self.d_out, int(max_batch), self.task, self.precision, int(seed),
                     beta1, beta2, eps, int(bool(wd_on_bias)), int(bool(fuse_optimizer)))
        drop = np.ascontiguousarray(dropout, dtype=np.float32)
        lr_ = np.ascontiguousarray(lr, dtype=np.float32)
        wd_ = np.ascontiguousarray(wd, dtype=np.float32)
        h = ctypes.c_void_p()
        self.d_emb = None
        if d_emb is None:
            _check(L.pack_create(ctypes.byref(cfg), _hptr(self.depth), _hptr(self.width), _hptr(drop), _hptr(lr_),
                                 _hptr(wd_), _stream_ptr(stream), ctypes.byref(h)))
        else:
            self.d_emb = np.ascontiguousarray(d_emb, dtype=np.int32)
            fr = np.ascontiguousarray(freq, dtype=np.float32)
            if self.d_emb.shape != (self.m,) or fr.size != self.d_in * int(np.sum(self.d_emb - 1)):
                raise ValueError("d_emb must hold m sizes and freq d_in (d_emb[i] - 1) values per member")
            _check(L.pack_create_emb(ctypes.byref(cfg), _hptr(self.depth), _hptr(self.width), _hptr(drop),
                                     _hptr(lr_), _hptr(wd_), _hptr(self.d_emb), _hptr(fr), _stream_ptr(stream),
                                     ctypes.byref(h)))
        self._h = h
        self._B = 0

    def close(self):
        if getattr(self, "_h", None):
            load_library().pack_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _y_dtype(self):
        return self.torch.float32 if self.task == REGRESSION else self.torch.int32

    def train_step(self, X, idx, y, step, loss_out=None, update=True):
        """X float32 [n, d_in], idx int32 [B] (one batch for every member) or
        [m, B] (a batch per member), y labels [n] (CUDA tensors); loss_out:
        optional float32 [m] CUDA tensor."""
        L = load_library()
        t = self.torch
        if idx.dim() == 2:
            if idx.shape[0] != self.m:
                raise ValueError("stacked idx must have one row per member")
            fn = L.pack_train_step_stacked if update else L.pack_forward_backward_stacked
            B = int(idx.shape[1])
        else:
            fn = L.pack_train_step if update else L.pack_forward_backward
            B = int(idx.shape[0])
        _check(fn(self._h, _dptr(X, t.float32), X.shape[0], _dptr(idx, t.int32), _dptr(y, self._y_dtype()),
                  B, int(step), _dptr(loss_out, t.float32)), self._h)
        self._B = B

    def forward_backward(self, X, idx, y, step, loss_out=None):
        self.train_step(X, idx, y, step, loss_out, update=False)

    def predict(self, X, out=None):
        t = self.torch
        if out is None:
            out = t.empty((self.m, X.shape[0], self.d_out), dtype=t.float32, device=X.device)
        _check(load_library().pack_predict(self._h, _dptr(X, t.float32), X.shape[0], _dptr(out, t.float32)), self._h)
        return out

    def set_active(self, active):
        a = np.ascontiguousarray(active, dtype=np.uint8)
        _check(load_library().pack_set_active(self._h, _hptr(a)), self._h)

    def set_muon(self, lr_muon, momentum=0.95, ns_steps=5):
        """Muon for the hidden-layer weights from the next step on."""
        lr = np.ascontiguousarray(lr_muon, dtype=np.float32)
        _check(load_library().pack_set_muon(self._h, _hptr(lr), float(momentum), int(ns_steps)), self._h)

    def muon_dir(self, member, layer):
        o, i = self.layer_shape(member, layer)
        out = np.zeros((o, i), dtype=np.float32)
        _check(load_library().pack_debug_muon_dir(self._h, int(member), int(layer), _hptr(out)), self._h)
        return out

    def get_active(self):
        a = np.zeros(self.m, dtype=np.uint8)
        _check(load_library().pack_get_active(self._h, _hptr(a)), self._h)
        return a

    def member_size(self, member):
        n = ctypes.c_int64()
        _check(load_library().pack_member_size(self._h, int(member), ctypes.byref(n)), self._h)
        return n.value

    def snapshot(self, member, out=None):
        """Member's parameter run (float32 CUDA tensor of member_size elements)."""
        t = self.torch
        if out is None:
            out = t.empty(self.member_size(member), dtype=t.float32, device="cuda")
        _check(load_library().pack_snapshot(self._h, int(member), _dptr(out, t.float32)), self._h)
        return out

    def restore(self, member, run):
        if run.numel() != self.member_size(member):
            raise ValueError("snapshot size does not match the member")
        _check(load_library().pack_restore(self._h, int(member), _dptr(run, self.torch.float32)), self._h)

    def layer_shape(self, member, layer):
        L, w = int(self.depth[member]), int(self.width[member])
        d0 = self.d_in * (int(self.d_emb[member]) if self.d_emb is not None else 1)
        return (self.d_out if layer == L else w), (d0 if layer == 0 else w)

    def emb(self, member, grads=False):
        """(w, b, alpha, beta) of a member's embeddings, or their gradients
        from the last step."""
        if self.d_emb is None:
            _check(load_library().pack_get_emb(self._h, 0, 0, None), self._h)
        d, n = int(self.d_emb[member]), self.d_in
        out = np.zeros(n * (4 * d - 2), dtype=np.float32)
        _check(load_library().pack_get_emb(self._h, int(member), int(bool(grads)), _hptr(out)), self._h)
        k = n * (d - 1)
        return (out[:k].reshape(n, d - 1), out[k:2 * k].reshape(n, d - 1), out[2 * k:2 * k + n * d].reshape(n, d),
                out[2 * k + n * d:].reshape(n, d))

    def set_emb(self, member, w, b, alpha, beta):
        if self.d_emb is None:
            _check(load_library().pack_set_emb(self._h, 0, None), self._h)
        d, n = int(self.d_emb[member]), self.d_in
        parts = [np.asarray(a, dtype=np.float32) for a in (w, b, alpha, beta)]
        if [p.size for p in parts] != [n * (d - 1), n * (d - 1), n * d, n * d]:
            raise ValueError("shape mismatch")
        flat = np.ascontiguousarray(np.concatenate([p.ravel() for p in parts]))
        _check(load_library().pack_set_emb(self._h, int(member), _hptr(flat)), self._h)

    def _valid(self, member, layer):
        return 0 <= member < self.m and 0 <= layer <= int(self.depth[member])

    def _two(self, fn, member, layer):
        if not self._valid(member, layer):   # let the library report the error
            _check(fn(self._h, int(member), int(layer), None, None), self._h)
        o, i = self.layer_shape(member, layer)
        W = np.zeros((o, i), dtype=np.float32)
        b = np.zeros(o, dtype=np.float32)
        _check(fn(self._h, member, layer, _hptr(W), _hptr(b)), self._h)
        return W, b

    def get_params(self, member, layer):
        return self._two(load_library().pack_get_params, member, layer)

    def get_grads(self, member, layer):
        return self._two(load_library().pack_get_grads, member, layer)

    def set_params(self, member, layer, W, b):
        if not self._valid(member, layer):
            _check(load_library().pack_set_params(self._h, int(member), int(layer), None, None), self._h)
        W = np.ascontiguousarray(W, dtype=np.float32)
        b = np.ascontiguousarray(b, dtype=np.float32)
        if W.shape != self.layer_shape(member, layer) or b.shape != (W.shape[0],):
            raise ValueError("shape mismatch")
        _check(load_library().pack_set_params(self._h, member, layer, _hptr(W), _hptr(b)), self._h)

    def logits(self, member):
        out = np.zeros((self._B, self.d_out), dtype=np.float32)
        _check(load_library().pack_get_logits(self._h, member, _hptr(out)), self._h)
        return out

    def debug_masks(self, member, layer, step, B):
        out = np.zeros((B, int(self.width[member])), dtype=np.uint8)
        _check(load_library().pack_debug_masks(self._h, member, layer, int(step), int(B), _hptr(out)), self._h)
        return out

    def debug_mask_arena(self, member, layer, B):
        """(keep [B, width] uint8, step) held in the bf16 mask arena."""
        out = np.zeros((B, int(self.width[member])), dtype=np.uint8)
        held = ctypes.c_int64(0)
        _check(load_library().pack_debug_mask_arena(self._h, member, layer, int(B), _hptr(out), ctypes.byref(held)),
               self._h)
        return out, held.value

    def debug_gemm_timeout(self, wait_s, poison=False):
        """Wait budget of the tensor-core launches; poison: one forward
        dependency that is never met (tests of the bounded waits)."""
        _check(load_library().pack_debug_gemm_timeout(self._h, float(wait_s), int(bool(poison))), self._h)

    def debug_bias_path(self, mode):
        """bf16: where the tensor-core weight-gradient products take the
        bias gradient from -- 1: column sums of dZ for every layer whose
        input width is a multiple of 256, 0: the bias column everywhere,
        -1: the pack's own choice."""
        _check(load_library().pack_debug_bias_path(self._h, int(mode)), self._h)

    def debug_activations(self, member, layer):
        out = np.zeros((self._B, int(self.width[member])), dtype=np.float32)
        _check(load_library().pack_debug_activations(self._h, member, layer, _hptr(out)), self._h)
        return out

    def profile_enable(self, on=True):
        _check(load_library().pack_profile_enable(self._h, int(bool(on))), self._h)

    def profile_read(self, reset=True):
        ms = np.zeros(len(PHASES), dtype=np.float64)
        n = np.zeros(len(PHASES), dtype=np.int64)
        _check(load_library().pack_profile_read(self._h, _hptr(ms), _hptr(n), int(bool(reset))), self._h)
        return {p: (float(ms[k]), int(n[k])) for k, p in enumerate(PHASES)}

    def launch_count(self):
        return int(load_library().pack_launch_count(self._h))

    def sizes(self):
        n = ctypes.c_int64()
        b = ctypes.c_int64()
        _check(load_library().pack_sizes(self._h, ctypes.byref(n), ctypes.byref(b)), self._h)
        return n.value, b.value


def debug_philox(ctr, key):
    """The device's Philox4x32-10 words [n, 4] for counters [n, 4], keys [n, 2]."""
    c = np.ascontiguousarray(np.atleast_2d(ctr), dtype=np.uint32)
    k = np.ascontiguousarray(np.atleast_2d(key), dtype=np.uint32)
    if c.shape[1] != 4 or k.shape != (c.shape[0], 2):
        raise ValueError("ctr must be [n, 4] and key [n, 2]")
    out = np.zeros((c.shape[0], 4), dtype=np.uint32)
    _check(load_library().pack_debug_philox(_hptr(c), _hptr(k), c.shape[0], _hptr(out)))
    return out


def select_greedy(preds, y, task, score="loss", m_ens=32, stream=None, static_scratch=False):
    """Greedy ensemble selection on the GPU.  preds float32 [P, N, d_out] and
    y [N] CUDA tensors.  Returns (selected indices, final score).
    static_scratch=True calls pack_select_greedy_static, the variant that
    allocates no device memory (its scratch is a fixed array in the library)."""
    import torch
    t = TASKS[task] if isinstance(task, str) else int(task)
    s = SCORES[score] if isinstance(score, str) else int(score)
    P, N, d_out = preds.shape
    ydt = torch.float32 if t == REGRESSION else torch.int32
    sel = np.zeros(m_ens, dtype=np.int32)
    n = ctypes.c_int32()
    fin = ctypes.c_double()
    fn = load_library().pack_select_greedy_static if static_scratch else load_library().pack_select_greedy
    _check(fn(_dptr(preds, torch.float32), P, N, d_out, _dptr(y, ydt), t, s, int(m_ens), _stream_ptr(stream),
              _hptr(sel), ctypes.byref(n), ctypes.byref(fin)))
    return sel[:n.value].copy(), fin.value


def _ocheck(status, handle):
    if status != TP_OK:
        msg = load_library().pack_online_last_error(handle)
        raise TabpackError(status, msg.decode() if msg else "")


class OnlineEnsemble:
    """Online ensemble of a Pack (Sec. 3.5) with ensemble and base-model
    early stopping (Sec. 3.6); see pack_online_create."""

    def __init__(self, pack, n_val, score="loss", m_ens=32, p_base=16, p_ens=32):
        L = load_library()
        self.pack = pack
        self.n_val = int(n_val)
        self.m_ens = int(m_ens)
        s = SCORES[score] if isinstance(score, str) else int(score)
        h = ctypes.c_void_p()
        _ocheck(L.pack_online_create(pack._h, self.n_val, s, self.m_ens, int(p_base), int(p_ens), ctypes.byref(h)),
                None)
        self._h = h

    def close(self):
        if getattr(self, "_h", None):
            load_library().pack_online_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def epoch(self, X_val, y_val):
        """End of an epoch; returns the stop flag."""
        t = self.pack.torch
        stop = ctypes.c_int32()
        _ocheck(load_library().pack_online_epoch(self._h, _dptr(X_val, t.float32), _dptr(y_val, self.pack._y_dtype()),
                                                 ctypes.byref(stop)), self._h)
        return bool(stop.value)

    def info(self):
        i = OnlineInfo()
        _ocheck(load_library().pack_online_info(self._h, ctypes.byref(i)), self._h)
        return {f: getattr(i, f) for f, _ in OnlineInfo._fields_}

    def members(self):
        m = self.pack.m
        sc, best = np.zeros(m), np.zeros(m)
        bad = np.zeros(m, dtype=np.int32)
        _ocheck(load_library().pack_online_members(self._h, _hptr(sc), _hptr(best), _hptr(bad)), self._h)
        return sc, best, bad

    def ensemble(self, which="best"):
        """(members, epochs, score) of the best or the last ensemble."""
        w = {"best": 0, "last": 1}[which]
        mem = np.zeros(self.m_ens, dtype=np.int32)
        ep = np.zeros(self.m_ens, dtype=np.int32)
        n = ctypes.c_int32()
        sc = ctypes.c_double()
        _ocheck(load_library().pack_online_ensemble(self._h, w, _hptr(mem), _hptr(ep), ctypes.byref(n),
                                                    ctypes.byref(sc)), self._h)
        return mem[:n.value].copy(), ep[:n.value].copy(), sc.value

    def snapshot(self, j):
        mem, _, _ = self.ensemble("best")
        t = self.pack.torch
        out = t.empty(self.pack.member_size(int(mem[j])), dtype=t.float32, device="cuda")
        _ocheck(load_library().pack_online_snapshot(self._h, int(j), _dptr(out, t.float32)), self._h)
        return out

    def predict(self, X, out=None):
        t = self.pack.torch
        if out is None:
            out = t.empty((X.shape[0], self.pack.d_out), dtype=t.float32, device=X.device)
        _ocheck(load_library().pack_online_predict(self._h, _dptr(X, t.float32), X.shape[0], _dptr(out, t.float32)),
                self._h)
        return out
