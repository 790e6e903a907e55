"""Pins of the oracle's Muon (Sec. 3.4 / App. F.1: Muon for the hidden-layer
weight matrices, AdamW for biases and the head; Jordan et al. 2024).

* The Newton-Schulz iteration is a polynomial in X X^T applied to X, so it
  keeps the singular vectors of U and maps each singular value s to q(s /
  ||U||_F), q being five compositions of p(x) = a x + b x^3 + c x^5: checked
  against numpy's SVD on wide, tall and square matrices.
* The optimizer step (momentum, Nesterov, the learning-rate adjustment, the
  decoupled weight decay) against torch.optim.Muon with its orthogonalizer
  replaced by the oracle's fp64 one (torch's own runs in bf16), and the
  biases and head against torch.optim.AdamW, over three steps.
"""
import numpy as np
import pytest

import oracle
from workloads import random_pack

A_, B_, C_ = 3.4445, -4.7750, 2.0315


def q5(x, steps=5):
    for _ in range(steps):
        x = A_ * x + B_ * x ** 3 + C_ * x ** 5
    return x


@pytest.mark.parametrize("shape", [(7, 19), (19, 7), (12, 12), (1, 5)])
def test_newton_schulz_maps_singular_values(shape):
    rng = np.random.default_rng(shape[0] * 31 + shape[1])
    U = rng.standard_normal(shape)
    O = oracle.newton_schulz(U, steps=5)
    P, s, Qt = np.linalg.svd(U, full_matrices=False)
    expect = P @ np.diag(q5(s / np.linalg.norm(U))) @ Qt
    np.testing.assert_allclose(O, expect, rtol=0, atol=1e-10)


def test_newton_schulz_transpose_scale_and_steps():
    rng = np.random.default_rng(4)
    U = rng.standard_normal((9, 23))
    O = oracle.newton_schulz(U)
    np.testing.assert_allclose(oracle.newton_schulz(U.T), O.T, atol=1e-12)
    np.testing.assert_allclose(oracle.newton_schulz(3.0 * U), O, atol=1e-12)
    # one step: a X + (b A + c A A) X with X = U / ||U||
    X = U / np.linalg.norm(U)
    G = X @ X.T
    np.testing.assert_allclose(oracle.newton_schulz(U, steps=1), A_ * X + (B_ * G + C_ * G @ G) @ X, atol=1e-13)
    # bf16 storage stays close to the exact iteration
    Ob = oracle.newton_schulz(U, bf16=True)
    assert np.max(np.abs(Ob - O)) / np.sqrt(np.mean(O ** 2)) < 0.1


@pytest.mark.parametrize("task,d_out", [("multiclass", 3), ("regression", 1)])
def test_muon_step_matches_torch_muon(task, d_out):
    torch = pytest.importorskip("torch")
    muon_mod = pytest.importorskip("torch.optim._muon")
    d_in, m, B = 6, 1, 24
    hp = random_pack(m, d_in, d_out, seed=12, width=(16, 32, 16), depth=(2, 2), dropout=(0.0, 0.0))
    lr_m = np.array([0.02])
    rng = np.random.default_rng(7)
    X = rng.standard_normal((60, d_in)).astype(np.float32)
    y = rng.integers(0, d_out, 60).astype(np.int32) if task == "multiclass" else rng.standard_normal(60).astype(np.float32)
    mk = lambda: oracle.OraclePack(d_in, d_out, task, hp["depth"], hp["width"], hp["dropout"], hp["lr"], hp["wd"], seed=3)
    pa, pb = mk(), mk()
    pa.set_muon(lr_m, momentum=0.95, ns_steps=5)
    L = int(hp["depth"][0])
    # torch twins of the parameters, fp64
    Ws, bs = [], []
    for l in range(L + 1):
        W, b = pa.get_params(0, l)
        Ws.append(torch.tensor(W, dtype=torch.float64, requires_grad=True))
        bs.append(torch.tensor(b, dtype=torch.float64, requires_grad=True))
    lr, wd = float(hp["lr"][0]), float(hp["wd"][0])
    opt_m = torch.optim.Muon(Ws[:L], lr=float(lr_m[0]), weight_decay=wd, momentum=0.95, nesterov=True, ns_steps=5)
    opt_a = torch.optim.AdamW(bs + [Ws[L]], lr=lr, weight_decay=wd, betas=(0.9, 0.999), eps=1e-8)
    saved = muon_mod._zeropower_via_newtonschulz
    muon_mod._zeropower_via_newtonschulz = lambda g, coeffs, steps, eps: torch.from_numpy(
        oracle.newton_schulz(g.detach().double().numpy(), steps=steps))
    try:
        for step in range(3):
            idx = rng.choice(60, B, replace=False).astype(np.int32)
            for l in range(L + 1):            # the twin holds the same parameters
                pb.set_params(0, l, Ws[l].detach().numpy(), bs[l].detach().numpy())
            pb.train_step(X, idx, y, step, update=False)
            pa.train_step(X, idx, y, step)
            for l in range(L + 1):
                gW, gb = pb.get_grads(0, l)
                Ws[l].grad = torch.tensor(gW, dtype=torch.float64)
                bs[l].grad = torch.tensor(gb, dtype=torch.float64)
            opt_m.step()
            opt_a.step()
            for l in range(L + 1):
                W, b = pa.get_params(0, l)
                np.testing.assert_allclose(W, Ws[l].detach().numpy(), rtol=0, atol=1e-12, err_msg=f"W{l} step {step}")
                np.testing.assert_allclose(b, bs[l].detach().numpy(), rtol=0, atol=1e-12, err_msg=f"b{l} step {step}")
    finally:
        muon_mod._zeropower_via_newtonschulz = saved
    # the direction the oracle applied last is its own Newton-Schulz output
    assert pa.muon_dir(0, 0).shape == Ws[0].shape
