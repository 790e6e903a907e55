"""Seeded synthetic workloads and hyperparameter sampling.

This module is shared by the tests, the benchmark and the smoke check.  It
holds no arithmetic of the method itself: it only draws inputs (feature
tables, labels from random teacher networks, batch index streams) and samples
each member's hyperparameters from the stated ranges (Sec. 3.7
"Hyperparameters": base-model hyperparameters are drawn at random from
user-defined spaces).

The five workloads stand in for the paper's benchmark datasets (17 tables,
10K to 1M+ rows, 8 to 900+ features; Appendix E, Table "dataset
properties"), which are not available here.  Seeds: data 0, hyperparameters
1, parameter init / dropout = the pack seed 2, batch shuffling 3.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch

SEED_DATA, SEED_HP, SEED_INIT, SEED_SHUFFLE = 0, 1, 2, 3


@dataclass(frozen=True)
class Workload:
    name: str
    task: str                 # "binary" | "multiclass" | "regression"
    n_train: int
    n_val: int
    d_in: int
    d_out: int
    m: int                    # members in the pack
    depth: tuple              # inclusive UniformInt range
    width: tuple              # (lo, hi, step): uniform over multiples of step
    dropout: tuple            # Uniform[lo, hi]
    lr: tuple = (1e-4, 3e-3)  # LogUniform
    wd: tuple = (1e-5, 1e-2)  # LogUniform
    batch: int = 256
    epochs: int = 1
    extra: dict = field(default_factory=dict)


WORKLOADS = {
    # binary, sign of a 2-layer ReLU teacher (width 32) with 5% label flips
    "tiny": Workload("tiny", "binary", 2048, 512, 8, 1, 8, (1, 3), (64, 256, 16), (0.0, 0.3),
                     batch=256, epochs=10),
    # regression, 8 Student-t(3) columns, 3-layer teacher (widths 64) + N(0, 0.1) noise
    "medium": Workload("medium", "regression", 100_000, 20_000, 64, 1, 32, (1, 4), (128, 1024, 64),
                       (0.0, 0.5), batch=512),
    # 10-class, 600 N(0,1) + 30 one-hot categoricals of cardinality 10
    "large": Workload("large", "multiclass", 700_000, 100_000, 900, 10, 64, (1, 4), (256, 1024, 128),
                      (0.0, 0.5), batch=1024),
    # many narrow members, binary labels from a random teacher
    "narrow": Workload("narrow", "binary", 300_000, 60_000, 128, 1, 256, (1, 3), (32, 256, 16),
                       (0.0, 0.3), batch=256),
    # wide members, regression target from a random teacher
    "wide": Workload("wide", "regression", 500_000, 100_000, 512, 1, 16, (4, 4), (1024, 2048, 256),
                     (0.0, 0.2), batch=2048),
}


def sample_hparams(wl: Workload, seed: int = SEED_HP, m: int | None = None) -> dict:
    """Per-member hyperparameters drawn from the workload's ranges."""
    m = wl.m if m is None else m
    rng = np.random.default_rng(seed)
    depth = rng.integers(wl.depth[0], wl.depth[1] + 1, size=m).astype(np.int32)
    lo, hi, step = wl.width
    width = (step * rng.integers(lo // step, hi // step + 1, size=m)).astype(np.int32)
    dropout = rng.uniform(wl.dropout[0], wl.dropout[1], size=m).astype(np.float32)
    lr = np.exp(rng.uniform(math.log(wl.lr[0]), math.log(wl.lr[1]), size=m)).astype(np.float32)
    wd = np.exp(rng.uniform(math.log(wl.wd[0]), math.log(wl.wd[1]), size=m)).astype(np.float32)
    return dict(depth=depth, width=width, dropout=dropout, lr=lr, wd=wd)


def _teacher(X: torch.Tensor, widths, gen: torch.Generator) -> torch.Tensor:
    """A random ReLU network with N(0, 1/fan_in) weights and zero biases."""
    h = X
    dims = [X.shape[1]] + list(widths)
    for li in range(len(dims) - 1):
        W = torch.randn(dims[li], dims[li + 1], generator=gen, device=X.device) / math.sqrt(dims[li])
        h = h @ W
        if li < len(dims) - 2:
            h = torch.relu(h)
    return h


def make_data(wl: Workload, device="cpu", seed: int = SEED_DATA, n_train: int | None = None,
              n_val: int | None = None) -> dict:
    """Feature table and labels, train and validation split, as torch tensors
    on `device`.  X is float32 [n, d_in]; y is int32 (classification) or
    float32 (regression)."""
    n_train = wl.n_train if n_train is None else n_train
    n_val = wl.n_val if n_val is None else n_val
    n = n_train + n_val
    dev = torch.device(device)
    gen = torch.Generator(device=dev)
    gen.manual_seed(seed)
    if wl.name == "large":
        num = torch.randn(n, 600, generator=gen, device=dev)
        cats = torch.randint(0, 10, (n, 30), generator=gen, device=dev)
        onehot = torch.zeros(n, 300, device=dev)
        onehot.scatter_(1, cats + 10 * torch.arange(30, device=dev), 1.0)
        X = torch.cat([num, onehot], dim=1)
    else:
        X = torch.randn(n, wl.d_in, generator=gen, device=dev)
        if wl.name == "medium":
            # Student-t with 3 degrees of freedom: z / sqrt(chi2_3 / 3)
            z = torch.randn(n, 8, generator=gen, device=dev)
            chi2 = (torch.randn(n, 8, 3, generator=gen, device=dev) ** 2).sum(-1)
            X[:, :8] = z / torch.sqrt(chi2 / 3.0)
    X = X.float().contiguous()
    if wl.name == "tiny":
        s = _teacher(X, [32, 1], gen)[:, 0]
        y = (s > 0).to(torch.int32)
        flip = torch.rand(n, generator=gen, device=dev) < 0.05
        y = torch.where(flip, 1 - y, y)
    elif wl.name == "medium":
        t = _teacher(X, [64, 64, 1], gen)[:, 0] + 0.1 * torch.randn(n, generator=gen, device=dev)
        mu, sd = t[:n_train].mean(), t[:n_train].std()
        y = ((t - mu) / sd).float()
    elif wl.name == "large":
        y = torch.argmax(_teacher(X, [64, 10], gen), dim=1).to(torch.int32)
    elif wl.name == "narrow":
        y = (_teacher(X, [64, 1], gen)[:, 0] > 0).to(torch.int32)
    else:  # wide
        t = _teacher(X, [64, 1], gen)[:, 0]
        mu, sd = t[:n_train].mean(), t[:n_train].std()
        y = ((t - mu) / sd).float()
    return dict(X_train=X[:n_train].contiguous(), y_train=y[:n_train].contiguous(),
                X_val=X[n_train:].contiguous(), y_val=y[n_train:].contiguous())


def batch_indices(n_train: int, batch: int, epoch: int, seed: int = SEED_SHUFFLE) -> list:
    """The row indices of each batch of one epoch (a seeded permutation cut
    into consecutive batches; the last batch may be short)."""
    rng = np.random.default_rng([seed, epoch])
    perm = rng.permutation(n_train).astype(np.int32)
    return [perm[s:s + batch] for s in range(0, n_train, batch)]


def random_pack(m, d_in, d_out, seed, depth=(1, 3), width=(16, 96, 16), dropout=(0.0, 0.4),
                lr=(1e-4, 3e-3), wd=(1e-5, 1e-2)) -> dict:
    """Small random pack shapes for tests."""
    wl = Workload("test", "binary", 0, 0, d_in, d_out, m, depth, width, dropout, lr, wd)
    return sample_hparams(wl, seed=seed, m=m)


def sample_emb(m, d_in, seed, d_emb=(8, 32, 4), sigma=(1e-2, 10.0)) -> dict:
    """Periodic-embedding hyperparameters of m members (App. "Feature
    Embeddings", TabPack-with-embeddings sampling space: d_emb UniformInt
    [8, 32] step 4, sigma LogUniform[1e-2, 10]) and the initial frequencies
    w ~ N(0, sigma) of each member, [d_in, d_emb - 1] row-major, member after
    member (float32 values, as the library takes them)."""
    rng = np.random.default_rng([seed, 7])
    lo, hi, step = d_emb
    d = rng.integers(0, (hi - lo) // step + 1, m) * step + lo
    s = np.exp(rng.uniform(np.log(sigma[0]), np.log(sigma[1]), m))
    freq = np.concatenate([rng.normal(0.0, s[i], d_in * (int(d[i]) - 1)) for i in range(m)] + [np.zeros(0)])
    return dict(d_emb=d.astype(np.int32), sigma=s, freq=freq.astype(np.float32))
