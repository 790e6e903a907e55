"""pack_select_greedy_static: greedy selection that allocates no device memory.

Some callers cannot allocate when they select (their device memory is fully
reserved by another framework's caching allocator, they run in a loop that
must not risk an out-of-memory failure or an allocator synchronisation, or
their runtime forbids allocation after start-up).  The variant serves them
from a fixed array of device memory defined in the library.  This file checks,
through the C ABI, that two calls in a row give the same selection as the
allocating entry point (indices identical, score within 1e-6 relative, the
bar of the other selection tests) and as the oracle's greedy selection on the
same candidates (Sec. 3.5; fp32 terms, the kernels' decision precision,
identical indices wherever the oracle's margin is not a near-tie), including
a ROC-AUC case sized near the array's limit; that a warmed-up call changes
neither the device's free memory nor torch's allocator statistics; and that a
problem too large for the array is refused with a clear error.  It runs last
(pytest collects files in name order) and also passes alone in a fresh
process.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tp():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_05380_gb300 import build
    build.build()
    import paper_2607_05380_gb300 as tpm
    tpm.load_library()
    return tpm


def _pool(task, P, N, C, seed):
    rng = np.random.default_rng(seed)
    if task == "multiclass":
        lg = rng.standard_normal((P, N, C)) * 1.5
        preds = np.exp(lg) / np.exp(lg).sum(-1, keepdims=True)
        y = rng.integers(0, C, N).astype(np.int32)
    elif task == "binary":
        preds = 1 / (1 + np.exp(-1.5 * rng.standard_normal((P, N, 1))))
        y = rng.integers(0, 2, N).astype(np.int32)
    else:
        y = rng.standard_normal(N).astype(np.float32)
        preds = y[None, :, None] + rng.standard_normal((P, N, 1)) * rng.uniform(0.5, 2, (P, 1, 1))
    return (torch.from_numpy(preds.astype(np.float32)).cuda(), torch.from_numpy(y).cuda())


def _oracle_agrees(preds, y, task, score, m_ens, sel):
    """The oracle's greedy selection on the same fp32 candidates gives the
    same indices up to its first near-tie (margin <= 1e-6 relative)."""
    import oracle
    osel, _, obest, ogap = oracle.greedy(preds.cpu().numpy(), y.cpu().numpy(), task, score, m_ens=m_ens,
                                         fp32_terms=True)
    k = 0
    while k < min(len(sel), len(osel)) and sel[k] == osel[k]:
        k += 1
    if k < max(len(sel), len(osel)):
        assert ogap[k] <= 1e-6 * max(1.0, abs(obest[k])), (list(sel), list(osel), ogap)


def test_two_calls_match_allocating_entry_point(tp):
    cases = [("multiclass", "loss", 48, 20000, 10, 16, 1), ("binary", "accuracy", 30, 3000, 1, 9, 2),
             ("regression", "rmse", 20, 7000, 1, 12, 3),
             # ROC-AUC near the 16 MiB limit: 80 candidates x 20000 rows need 16.2 MB with the sort buffers
             ("binary", "auc", 80, 20000, 1, 10, 4)]
    for task, score, P, N, C, m_ens, seed in cases:
        preds, y = _pool(task, P, N, C, seed)
        ref_sel, ref_fin = tp.select_greedy(preds, y, task, score, m_ens=m_ens)
        got_sel, got_fin = tp.select_greedy(preds, y, task, score, m_ens=m_ens, static_scratch=True)
        assert list(got_sel) == list(ref_sel), (task, score)
        assert abs(got_fin - ref_fin) <= 1e-6 * max(1.0, abs(ref_fin)), (task, score)
        _oracle_agrees(preds, y, task, score, m_ens, list(got_sel))
    # the same problem again right after a different one: no stale state
    preds, y = _pool("multiclass", 48, 20000, 10, 1)
    ref_sel, ref_fin = tp.select_greedy(preds, y, "multiclass", "loss", m_ens=16)
    got_sel, got_fin = tp.select_greedy(preds, y, "multiclass", "loss", m_ens=16, static_scratch=True)
    assert list(got_sel) == list(ref_sel)
    assert abs(got_fin - ref_fin) <= 1e-6 * max(1.0, abs(ref_fin))


def test_allocates_nothing(tp):
    """After a warm-up call, further calls change neither the device's free
    memory nor torch's allocator statistics."""
    preds, y = _pool("binary", 64, 20000, 1, 5)
    for score in ("auc", "loss"):    # warm-up: every kernel of both scores loaded
        tp.select_greedy(preds, y, "binary", score, m_ens=8, static_scratch=True)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    alloc0, res0 = torch.cuda.memory_allocated(), torch.cuda.memory_reserved()
    for score in ("auc", "loss", "auc"):
        tp.select_greedy(preds, y, "binary", score, m_ens=8, static_scratch=True)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0
    assert (torch.cuda.memory_allocated(), torch.cuda.memory_reserved()) == (alloc0, res0)


def test_too_large_is_refused(tp):
    P, N, C = 4, 300_000, 10          # 24 MB of running sum alone
    preds = torch.zeros(P, N, C, dtype=torch.float32, device="cuda")
    y = torch.zeros(N, dtype=torch.int32, device="cuda")
    with pytest.raises(tp.TabpackError) as ei:
        tp.select_greedy(preds, y, "multiclass", "loss", m_ens=2, static_scratch=True)
    assert ei.value.status == tp.TP_EINVAL
    assert "scratch" in str(ei.value)
    # ROC-AUC's sort buffers count: 90 candidates x 20000 rows need 18 MB
    preds, y = _pool("binary", 90, 20000, 1, 6)
    with pytest.raises(tp.TabpackError) as ei:
        tp.select_greedy(preds, y, "binary", "auc", m_ens=2, static_scratch=True)
    assert ei.value.status == tp.TP_EINVAL and "ROC-AUC" in str(ei.value)
