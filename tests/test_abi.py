"""The C-ABI library loads on a host without a GPU and exports every entry
point declared in include/tabpack.h (no compute calls here)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib_path():
    from paper_2607_05380_gb300 import build
    return build.build()


def declared_functions():
    names = []
    for f in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if not f.endswith(".h"):
            continue
        src = open(os.path.join(ROOT, "include", f)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names += re.findall(r"^\s*(?:[\w\s\*]+?)\b(\w+)\s*\([^;{]*\)\s*;", src, flags=re.M)
    return sorted(set(n for n in names if n.startswith("pack_")))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("pack_create", "pack_train_step", "pack_predict", "pack_select_greedy", "pack_destroy"):
        assert n in names


def test_library_exports_every_declared_symbol(lib_path):
    lib = ctypes.CDLL(lib_path)
    for n in declared_functions():
        assert hasattr(lib, n), n
    out = subprocess.run(["nm", "-D", "--defined-only", lib_path], capture_output=True, text=True).stdout
    exported = set(line.split()[-1] for line in out.splitlines() if line.strip())
    assert set(declared_functions()) <= exported


def test_binding_lists_every_symbol(lib_path):
    import paper_2607_05380_gb300 as tp
    assert sorted(tp.SYMBOLS) == declared_functions()
    tp.load_library()


def test_create_without_gpu_fails_cleanly(lib_path):
    """On a host without a GPU pack_create reports an error status, it does
    not crash and does not fall back to the CPU."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("host has a GPU")
    import numpy as np
    import paper_2607_05380_gb300 as tp
    L = tp.load_library()
    cfg = tp.Config(1, 4, 1, 16, 0, 0, 1, 0.9, 0.999, 1e-8, 1)
    arr = lambda v, dt: np.array(v, dtype=dt)
    d, w, p, lr, wd = arr([1], np.int32), arr([16], np.int32), arr([0.1], np.float32), arr([1e-3], np.float32), arr([0.0], np.float32)
    h = ctypes.c_void_p()
    st = L.pack_create(ctypes.byref(cfg), tp._hptr(d), tp._hptr(w), tp._hptr(p), tp._hptr(lr), tp._hptr(wd), None,
                       ctypes.byref(h))
    assert st in (tp.TP_ECUDA, tp.TP_ENOTSUP)
    assert not h.value
    assert L.pack_last_error(None)


def test_invalid_configs_rejected_before_any_gpu_call(lib_path):
    import numpy as np
    import paper_2607_05380_gb300 as tp
    L = tp.load_library()
    arr = lambda v, dt: np.array(v, dtype=dt)
    base = dict(depth=[1], width=[16], drop=[0.1])
    cases = [
        (tp.Config(1, 4, 1, 16, 0, 0, 1, 0.9, 0.999, 1e-8, 1), [1], [24], [0.1]),   # width not multiple of 16
        (tp.Config(1, 4, 1, 16, 0, 0, 1, 0.9, 0.999, 1e-8, 1), [0], [16], [0.1]),   # depth 0
        (tp.Config(1, 4, 1, 16, 0, 0, 1, 0.9, 0.999, 1e-8, 1), [1], [16], [1.0]),   # dropout 1
        (tp.Config(1, 4, 3, 16, 0, 0, 1, 0.9, 0.999, 1e-8, 1), [1], [16], [0.1]),   # binary with d_out 3
        (tp.Config(0, 4, 1, 16, 0, 0, 1, 0.9, 0.999, 1e-8, 1), [1], [16], [0.1]),   # m = 0
        (tp.Config(1, 4, 40, 16, 1, 0, 1, 0.9, 0.999, 1e-8, 1), [1], [16], [0.1]),  # too many classes
    ]
    for cfg, d, w, p in cases:
        h = ctypes.c_void_p()
        st = L.pack_create(ctypes.byref(cfg), tp._hptr(arr(d, np.int32)), tp._hptr(arr(w, np.int32)),
                           tp._hptr(arr(p, np.float32)), tp._hptr(arr([1e-3], np.float32)),
                           tp._hptr(arr([0.0], np.float32)), None, ctypes.byref(h))
        assert st == tp.TP_EINVAL, (cfg.m, d, w, p)
        assert not h.value


def test_embedding_entry_points_reject_bad_arguments_without_a_gpu(lib_path):
    """pack_create_emb checks the embedding sizes and pointers before any GPU
    call; the embedding accessors reject a NULL pack."""
    import numpy as np
    import paper_2607_05380_gb300 as tp
    L = tp.load_library()
    arr = lambda v, dt: np.array(v, dtype=dt)
    cfg = tp.Config(2, 4, 1, 16, 0, 0, 1, 0.9, 0.999, 1e-8, 1)
    d, w, p = arr([1, 2], np.int32), arr([16, 32], np.int32), arr([0.1, 0.0], np.float32)
    lr, wd = arr([1e-3, 1e-3], np.float32), arr([0.0, 0.0], np.float32)
    freq = arr(np.zeros(4 * 70), np.float32)
    for d_emb, fr in (([0, 4], freq), ([4, 65], freq), ([4, 4], None), (None, freq)):
        h = ctypes.c_void_p()
        de = None if d_emb is None else tp._hptr(arr(d_emb, np.int32))
        st = L.pack_create_emb(ctypes.byref(cfg), tp._hptr(d), tp._hptr(w), tp._hptr(p), tp._hptr(lr), tp._hptr(wd),
                               de, None if fr is None else tp._hptr(fr), None, ctypes.byref(h))
        assert st == tp.TP_EINVAL, d_emb
        assert not h.value
    # a bad width is still caught with valid embedding sizes
    h = ctypes.c_void_p()
    st = L.pack_create_emb(ctypes.byref(cfg), tp._hptr(d), tp._hptr(arr([16, 24], np.int32)), tp._hptr(p),
                           tp._hptr(lr), tp._hptr(wd), tp._hptr(arr([4, 4], np.int32)), tp._hptr(freq), None,
                           ctypes.byref(h))
    assert st == tp.TP_EINVAL and not h.value
    out = arr(np.zeros(64), np.float32)
    n = ctypes.c_int32()
    assert L.pack_get_emb(None, 0, 0, tp._hptr(out)) == tp.TP_EINVAL
    assert L.pack_set_emb(None, 0, tp._hptr(out)) == tp.TP_EINVAL
    assert L.pack_member_emb(None, 0, ctypes.byref(n)) == tp.TP_EINVAL


def test_debug_hooks_reject_a_null_pack_without_a_gpu(lib_path):
    """The tensor-core debug hooks check their pack before any GPU call."""
    import paper_2607_05380_gb300 as tp
    L = tp.load_library()
    assert L.pack_debug_bias_path(None, 1) == tp.TP_EINVAL
    assert L.pack_debug_bias_path(None, -1) == tp.TP_EINVAL
    assert L.pack_debug_gemm_timeout(None, 1.0, 0) == tp.TP_EINVAL
    assert L.pack_last_error(None)
