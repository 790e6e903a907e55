"""Failure detection of the tensor-core products, on the GPU, without a
fault: a bounded wait is made to run out and the library must report it as
a status, leaving the device usable.

The test makes one forward tile wait for a dependency count its launch
never reaches (pack_debug_gemm_timeout).  That tile's producer waits before
it issues any copy, gives up after the budget, raises its CTA's abort flag
and records site 3; the CTA's MMA and epilogue roles see the flag in their
own bounded waits, the CTA lets its issued copies and MMAs finish, frees its
tensor memory and exits; CTAs whose tiles read that tile's output give up
the same way.  The pack is small (single-CTA tiles).  The next
synchronising call must return TP_ETIMEOUT naming the site, and a fresh
pack on the same device must then pass one step at the parity bars.
"""
import time

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from parity import Oracles, compare_step  # noqa: E402
from workloads import random_pack  # noqa: E402

DEV = "cuda"


@pytest.fixture(scope="module")
def tp():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2607_05380_gb300 import build
    build.build()
    import paper_2607_05380_gb300 as tpm
    tpm.load_library()
    return tpm


def _data(n, d_in, d_out, seed):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((n, d_in)).astype(np.float32)
    y = rng.integers(0, d_out, n).astype(np.int32)
    return X, y


def test_gemm_wait_runs_out(tp):
    d_in, d_out, m, B = 24, 3, 4, 256
    hp = random_pack(m, d_in, d_out, seed=61, width=(32, 96, 16), depth=(2, 3))
    X, y = _data(400, d_in, d_out, 1)
    idx = np.random.default_rng(2).choice(400, B, replace=False).astype(np.int32)
    Xd, yd, idxd = (torch.from_numpy(a).to(DEV) for a in (X, y, idx))
    loss = torch.zeros(m, dtype=torch.float32, device=DEV)

    pk = tp.Pack(d_in, d_out, "multiclass", hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"],
                 max_batch=B, seed=2, precision="bf16")
    pk.debug_gemm_timeout(0.3, poison=True)
    t0 = time.perf_counter()
    pk.forward_backward(Xd, idxd, yd, 1, loss)
    with pytest.raises(tp.TabpackError) as ei:
        pk.get_grads(0, 0)
    assert ei.value.status == tp.TP_ETIMEOUT, ei.value
    assert "wait site 3" in str(ei.value), ei.value
    assert time.perf_counter() - t0 < 30
    pk.close()

    # the device is still usable: a fresh pack passes one step at the parity bars
    pk2 = tp.Pack(d_in, d_out, "multiclass", hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"],
                  max_batch=B, seed=2, precision="bf16")
    orc = Oracles("bf16", d_in, d_out, "multiclass", hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"],
                  seed=2)
    pk2.forward_backward(Xd, idxd, yd, 1, loss)
    orc.train_step(X, idx, y, 1, update=False)
    problems = compare_step(pk2, orc, hp, "bf16", loss.cpu().numpy())
    assert not problems, problems
    pk2.close()


def test_timeout_budget_is_checked(tp):
    hp = random_pack(2, 8, 1, seed=3, depth=(2, 2))
    pk = tp.Pack(8, 1, "regression", hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"], max_batch=128,
                 seed=2, precision="bf16")
    with pytest.raises(tp.TabpackError) as ei:
        pk.debug_gemm_timeout(0.0)
    assert ei.value.status == tp.TP_EINVAL
    pk.close()
    pk = tp.Pack(8, 1, "regression", hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"], max_batch=128,
                 seed=2, precision="fp32")
    with pytest.raises(tp.TabpackError) as ei:
        pk.debug_gemm_timeout(1.0)
    assert ei.value.status == tp.TP_ESTATE
    pk.close()
