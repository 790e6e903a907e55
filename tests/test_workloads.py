"""The seeded input recipes: embedding hyperparameters drawn from the
paper's TabPack-with-embeddings sampling space (App. "Feature Embeddings":
d_emb UniformInt[8, 32] step 4, sigma LogUniform[1e-2, 10], w ~ N(0, sigma),
b = alpha = beta = 0 at the start), reproducibly."""
import numpy as np

from workloads import sample_emb


def test_embedding_sizes_and_scales_in_the_stated_space():
    e = sample_emb(4000, 3, seed=1)
    d, s = e["d_emb"], e["sigma"]
    assert set(np.unique(d).tolist()) == set(range(8, 33, 4))        # every size of the grid occurs
    assert s.min() >= 1e-2 and s.max() <= 10.0
    # log-uniform: log10(sigma) uniform on [-2, 1] (mean -0.5, variance 0.75)
    ls = np.log10(s)
    assert abs(ls.mean() + 0.5) < 0.05 and abs(ls.var() - 0.75) < 0.05


def test_frequencies_layout_and_scale():
    d_in = 200
    e = sample_emb(12, d_in, seed=2)
    d, s, f = e["d_emb"], e["sigma"], e["freq"]
    assert f.dtype == np.float32 and f.size == d_in * int(np.sum(d - 1))
    off = 0
    for i in range(12):   # member after member, [d_in, d_emb - 1] each, spread ~ sigma_i
        n = d_in * (int(d[i]) - 1)
        block = f[off:off + n].astype(np.float64)
        assert abs(block.std() / s[i] - 1.0) < 0.1, i
        off += n


def test_reproducible_and_seed_dependent():
    a, b, c = sample_emb(8, 5, seed=3), sample_emb(8, 5, seed=3), sample_emb(8, 5, seed=4)
    assert all(np.array_equal(a[k], b[k]) for k in a)
    assert not np.array_equal(a["freq"], c["freq"]) or not np.array_equal(a["d_emb"], c["d_emb"])
    one = sample_emb(3, 4, seed=1, d_emb=(1, 1, 1))   # d_emb = 1: no frequencies at all
    assert one["freq"].size == 0 and one["d_emb"].tolist() == [1, 1, 1]
