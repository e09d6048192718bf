"""The seeded synthetic inputs follow their stated recipe (CPU only).

Keys, values and queries stand in for the long-context workloads of the
paper's Sec. 5.1.  These tests check the properties each recipe promises, so
that the parity and benchmark inputs are what the documentation says:
  - every tensor is bf16-representable (the GPU and the oracle see the same values);
  - "outlier" keys: N(0, 1) with exactly 4 channels scaled by 6;
  - "logscale" keys: per-channel scale in [0.5, 4], log-uniform;
  - "mixture" keys: 16 orthonormal mean directions of norm sqrt(d), noise 0.5 per coordinate;
  - values N(0, 1);
  - queries: norm near sqrt(d (1 + 0.3^2)), aimed at the candidate pool (all rows, a
    fixed 5% hot set, or the rows of 2 fixed mixture components);
  - the same seed gives the same bytes, another seed does not.
"""
import numpy as np

from paper_2606_01563_gb300.inputs import WORKLOADS, Generator, Geometry, Workload, bf16_round


def _is_bf16(x):
    return np.array_equal(x, bf16_round(x))


def _aim(Q, K):
    """For each query row, the key row with the largest dot product."""
    return np.argmax(Q.reshape(-1, Q.shape[-1]) @ K.T, axis=1)


def test_bf16_and_determinism():
    wl = WORKLOADS["tiny_d64_t1k"]
    a, b, c = Generator(wl, seed=0), Generator(wl, seed=0), Generator(wl, seed=1)
    A, B, C = a.prefill(), b.prefill(), c.prefill()
    for x, y, z in zip(A, B, C):
        assert _is_bf16(x)
        assert np.array_equal(x, y)
        assert not np.array_equal(x, z)
    qa, qb = a.decode(4), b.decode(4)
    for x, y in zip(qa, qb):
        assert _is_bf16(x) and np.array_equal(x, y)
    G = wl.geom
    assert qa[0].shape == (4, G.batch, G.n_q_heads, G.head_dim)
    assert qa[1].shape == qa[2].shape == (4, G.batch, G.n_kv_heads, G.head_dim)


def test_outlier_keys_and_values():
    wl = Workload("o", Geometry(1, 2, 2, 64), 8192, 128, 16, "outlier")
    gen = Generator(wl, seed=3)
    K, V, Q = gen.prefill()
    for u in range(2):
        scale = gen._params[u]["scale"]
        assert np.count_nonzero(scale == 6.0) == 4 and np.count_nonzero(scale == 1.0) == 60
        np.testing.assert_allclose(K[0, u].std(axis=0), scale, rtol=0.05)
        assert abs(V[0, u].mean()) < 0.02 and abs(V[0, u].std() - 1.0) < 0.02


def test_logscale_keys_and_hot_queries():
    wl = Workload("l", Geometry(1, 2, 4, 128), 8192, 512, 32, "logscale")
    gen = Generator(wl, seed=5)
    K, V, Q = gen.prefill()
    d = 128
    for u in range(2):
        p = gen._params[u]
        scale = p["scale"]
        assert scale.min() >= 0.5 and scale.max() <= 4.0
        # log-uniform on [log 0.5, log 4]: mean of log scale near the midpoint
        assert abs(np.log(scale).mean() - 0.5 * (np.log(0.5) + np.log(4.0))) < 0.2
        np.testing.assert_allclose(K[0, u].std(axis=0), scale, rtol=0.06)
        hot = p["hot"]
        assert len(hot) == wl.T // 20 and len(np.unique(hot)) == len(hot) and hot.max() < wl.T
        q = Q[0, u].reshape(-1, d)
        norms = np.linalg.norm(q, axis=1)
        assert abs(np.median(norms) / np.sqrt(d * (1 + 0.3 ** 2)) - 1) < 0.1
        # each window query is built from 3 hot keys: its best-matching key is hot
        frac_hot = np.isin(_aim(q, K[0, u]), hot).mean()
        assert frac_hot > 0.9, frac_hot


def test_mixture_keys_and_component_queries():
    wl = Workload("m", Geometry(1, 2, 4, 128), 8192, 128, 64, "mixture")
    gen = Generator(wl, seed=7)
    K, V, Q = gen.prefill()
    d = 128
    for u in range(2):
        p = gen._params[u]
        means = p["means"]
        np.testing.assert_allclose(means @ means.T, d * np.eye(16), atol=1e-9)
        comp = gen._comp[u]
        assert set(np.unique(comp)) == set(range(16))
        noise = K[0, u] - means[comp]
        assert abs(noise.std() - 0.5) < 0.01
        hot_rows = np.nonzero(np.isin(comp, p["hot_comps"]))[0]
        q = Q[0, u].reshape(-1, d)
        frac_hot = np.isin(_aim(q, K[0, u]), hot_rows).mean()
        assert frac_hot > 0.9, frac_hot
        # keys of the other 14 components lie nearly orthogonal to the queries' directions
        cold = ~np.isin(comp, p["hot_comps"])
        hot_dir = means[p["hot_comps"]].sum(axis=0)
        cos = (K[0, u][cold] @ hot_dir) / (np.linalg.norm(K[0, u][cold], axis=1) * np.linalg.norm(hot_dir))
        assert np.abs(cos).mean() < 0.1


def test_bench_workloads_match_their_configurations():
    wl = WORKLOADS["llama8b_layer_t8k"]
    g = wl.geom
    assert (g.batch, g.n_kv_heads, g.group, g.head_dim) == (1, 8, 4, 128)
    assert (wl.T, wl.budget, wl.window, wl.decode_steps, wl.key_dist) == (8192, 512, 32, 256, "logscale")
    wl = WORKLOADS["qwen4b_t32k"]
    g = wl.geom
    assert (g.batch, g.n_kv_heads, g.group, g.head_dim) == (4, 8, 4, 128)
    assert (wl.T, wl.budget, wl.window) == (32768, 1024, 32) and wl.extra["budgets"] == (128, 256, 1024)
    wl = WORKLOADS["llama8b_t128k"]
    g = wl.geom
    assert (g.batch, g.n_kv_heads, g.group, g.head_dim) == (1, 8, 4, 128)
    assert (wl.T, wl.budget, wl.window, wl.key_dist, wl.evict_every) == (131072, 128, 64, "mixture", 64)
    wl = WORKLOADS["tiny_d64_t1k"]
    g = wl.geom
    assert (g.batch, g.n_kv_heads, g.group, g.head_dim) == (1, 2, 2, 64)
    assert (wl.T, wl.budget, wl.window, wl.decode_steps, wl.key_dist) == (1024, 128, 16, 16, "outlier")


# ---------------------------------------------------------------------------
# TorchGenerator: the same recipes drawn with torch (here on the CPU; the
# bench draws the multi-layer prompts on the GPU with the same code)
# ---------------------------------------------------------------------------
def _torch_unit(wl, seed=0, layer=0, T=None, steps=4):
    import torch  # noqa: F401
    from paper_2606_01563_gb300.inputs import TorchGenerator
    gen = TorchGenerator(wl, seed=seed, layer=layer)
    K, V, Q = gen.prefill(T)
    q, kn, vn = gen.decode(steps)
    return gen, [x.float().numpy() for x in (K, V, Q, q, kn, vn)]


def test_torch_generator_shapes_bf16_determinism():
    wl = WORKLOADS["tiny_d64_t1k"]
    _, A = _torch_unit(wl, seed=0, layer=1)
    _, B = _torch_unit(wl, seed=0, layer=1)
    _, C = _torch_unit(wl, seed=0, layer=2)
    G = wl.geom
    shapes = [(1, 2, 1024, 64), (1, 2, 1024, 64), (1, 2, 2, 16, 64), (4, 1, 4, 64), (4, 1, 2, 64), (4, 1, 2, 64)]
    for x, y, z, shp in zip(A, B, C, shapes):
        assert x.shape == shp and _is_bf16(x)
        assert np.array_equal(x, y)
        assert not np.array_equal(x, z)
    assert G.n_q_heads == 4


def test_torch_generator_logscale_recipe():
    wl = Workload("l", Geometry(1, 2, 4, 128), 8192, 512, 32, "logscale")
    gen, (K, V, Q, q, kn, vn) = _torch_unit(wl, seed=5, steps=64)
    d = 128
    for u in range(2):
        scale = gen.scale[u].numpy()
        assert scale.min() >= 0.5 and scale.max() <= 4.0
        assert abs(np.log(scale).mean() - 0.5 * (np.log(0.5) + np.log(4.0))) < 0.2
        np.testing.assert_allclose(K[0, u].std(axis=0), scale, rtol=0.06)
        assert abs(V[0, u].std() - 1.0) < 0.02
        hot = gen._pool[u].numpy()
        assert len(hot) == wl.T // 20 and len(np.unique(hot)) == len(hot)
        for qq in (Q[0, u].reshape(-1, d), q[:, 0, 4 * u:4 * u + 4].reshape(-1, d)):
            norms = np.linalg.norm(qq, axis=1)
            assert abs(np.median(norms) / np.sqrt(d * (1 + 0.3 ** 2)) - 1) < 0.1
            assert np.isin(_aim(qq, K[0, u]), hot).mean() > 0.9
        np.testing.assert_allclose(kn[:, 0, u].std(axis=0).mean(), np.sqrt((scale ** 2).mean()), rtol=0.25)


def test_torch_generator_mixture_recipe():
    wl = Workload("m", Geometry(1, 2, 4, 128), 8192, 128, 64, "mixture")
    gen, (K, V, Q, q, kn, vn) = _torch_unit(wl, seed=7)
    d = 128
    for u in range(2):
        means = gen.means[u].double().numpy()
        np.testing.assert_allclose(means @ means.T, d * np.eye(16), atol=1e-4)
        hot_comps = gen.hot_comps[u].numpy()
        assert len(set(hot_comps)) == 2
        # every key is a component mean plus N(0, 0.5^2) noise: the nearest mean explains it
        dist = ((K[0, u][:, None, :] - means[None].astype(np.float32)) ** 2).sum(-1)
        comp = dist.argmin(1)
        assert abs((K[0, u] - means[comp]).std() - 0.5) < 0.01
        hot_rows = np.nonzero(np.isin(comp, hot_comps))[0]
        assert np.array_equal(hot_rows, gen._pool[u].numpy())
        assert np.isin(_aim(Q[0, u].reshape(-1, d), K[0, u]), hot_rows).mean() > 0.9
