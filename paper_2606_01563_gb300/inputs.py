"""Seeded synthetic inputs shared by the tests, the benchmark and the smoke check.

This module only draws random numbers and rounds them to bf16; it holds none
of MomentKV's arithmetic, and both the CUDA path and the fp64 oracle consume
its arrays.  Distributions stand in for the long-context LLM workloads the
paper evaluates on (LongBench, RULER on Llama-3.1-8B and Qwen3-4B, Sec. 5.1),
whose data and weights are not used here.

Recipes (one numpy PCG64 stream per seed):
  keys "outlier":  N(0,1) with 4 random channels scaled x6.
  keys "logscale": N(0,1) times a per-channel scale drawn LogUniform(0.5, 4).
  keys "mixture":  16-component Gaussian mixture in R^d; component means are
                   orthonormal directions (QR of a Gaussian d x 16 matrix)
                   scaled to norm sqrt(d), uniform weights, within-component
                   noise N(0, 0.5^2) per coordinate.
  values:          N(0,1).
  queries:         u = sum of 3 key rows drawn from a candidate pool,
                   q = sqrt(d) u / ||u|| + N(0, 0.3^2) noise.  The pool is all
                   rows ("outlier"), a fixed random 5% of rows ("logscale"),
                   or the rows of 2 fixed components ("mixture").
Everything is rounded to bf16 (round to nearest even) before use.
Generator draws with numpy on the host; TorchGenerator draws the same
recipes with torch on a device, for the multi-layer workloads.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch


def bf16_round(x) -> np.ndarray:
    """Round to the nearest bf16 value; returned as float32 (exact)."""
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32))
    return t.to(torch.bfloat16).to(torch.float32).numpy()


def to_bf16_tensor(x) -> torch.Tensor:
    """float array -> torch.bfloat16 CPU tensor (round to nearest even)."""
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).to(torch.bfloat16)


@dataclass
class Geometry:
    batch: int
    n_kv_heads: int
    group: int
    head_dim: int

    @property
    def n_q_heads(self):
        return self.n_kv_heads * self.group


@dataclass
class Workload:
    name: str
    geom: Geometry
    T: int
    budget: int
    window: int
    key_dist: str
    decode_steps: int = 16
    evict_every: int = 0
    n_layers: int = 1
    sink: int = 1
    keep_window: int = 1
    pool: int = 1
    extra: dict = field(default_factory=dict)


WORKLOADS = {
    # tiny parity case: 1 layer, b=1, 2 KV heads x 2, d=64, T=1024, B=128, w=16
    "tiny_d64_t1k": Workload("tiny_d64_t1k", Geometry(1, 2, 2, 64), 1024, 128, 16,
                             "outlier", decode_steps=16),
    # Llama-3.1-8B attention geometry, one layer, T=8192, B=512, w=32, 256 decode steps
    "llama8b_layer_t8k": Workload("llama8b_layer_t8k", Geometry(1, 8, 4, 128), 8192, 512, 32,
                                  "logscale", decode_steps=256),
    # Qwen3-4B geometry, 36 layers, batch 4, T=32768, B in {128,256,1024}, w=32, 512 steps
    "qwen4b_t32k": Workload("qwen4b_t32k", Geometry(4, 8, 4, 128), 32768, 1024, 32,
                            "logscale", decode_steps=512, n_layers=36,
                            extra={"budgets": (128, 256, 1024)}),
    # Llama-3.1-8B geometry, 32 layers, T=131072, B=128, w=64, evict every 64 tokens
    "llama8b_t128k": Workload("llama8b_t128k", Geometry(1, 8, 4, 128), 131072, 128, 64,
                              "mixture", decode_steps=1024, evict_every=64, n_layers=32),
}

DECODE_SWEEP = {"batch": (1, 8, 32, 64), "budget": (256, 1024, 4096)}


class Generator:
    """Draws one workload's tensors.  Each (layer, batch, kv head) slab gets
    its own key distribution parameters and query pool."""

    def __init__(self, wl: Workload, seed: int = 0, layer: int = 0):
        self.wl = wl
        self.rng = np.random.default_rng(seed + 1000003 * layer)
        g = wl.geom
        d = g.head_dim
        self.units = g.batch * g.n_kv_heads
        self._params = []
        for _ in range(self.units):
            p = {}
            if wl.key_dist == "outlier":
                p["scale"] = np.ones(d)
                p["scale"][self.rng.choice(d, 4, replace=False)] = 6.0
            elif wl.key_dist == "logscale":
                p["scale"] = np.exp(self.rng.uniform(np.log(0.5), np.log(4.0), d))
            elif wl.key_dist == "mixture":
                A = self.rng.standard_normal((d, 16))
                Qm, _ = np.linalg.qr(A)
                p["means"] = Qm.T * np.sqrt(d)          # [16, d]
                p["hot_comps"] = self.rng.choice(16, 2, replace=False)
            else:
                raise ValueError(wl.key_dist)
            self._params.append(p)
        self._comp = [None] * self.units

    # -- keys / values -----------------------------------------------------
    def _keys(self, u, n, record=False):
        p = self._params[u]
        d = self.wl.geom.head_dim
        if "scale" in p:
            return self.rng.standard_normal((n, d)) * p["scale"]
        comp = self.rng.integers(0, 16, n)
        if record:
            self._comp[u] = comp
        return p["means"][comp] + 0.5 * self.rng.standard_normal((n, d))

    def _query_pool(self, u, T):
        p = self._params[u]
        if self.wl.key_dist == "outlier":
            return None
        if self.wl.key_dist == "logscale":
            if "hot" not in p or p["hot_T"] != T:
                p["hot"] = np.sort(self.rng.choice(T, max(3, T // 20), replace=False))
                p["hot_T"] = T
            return p["hot"]
        comp = self._comp[u]
        return np.nonzero(np.isin(comp, p["hot_comps"]))[0]

    def _queries(self, K, pool, n):
        d = K.shape[1]
        rows = (self.rng.integers(0, K.shape[0], (n, 3)) if pool is None
                else pool[self.rng.integers(0, len(pool), (n, 3))])
        u = K[rows].sum(axis=1)
        u = np.sqrt(d) * u / np.linalg.norm(u, axis=1, keepdims=True)
        return u + 0.3 * self.rng.standard_normal((n, d))

    def prefill(self, T=None):
        """K, V [b, Hkv, T, d], Q_obs [b, Hkv, g, w, d]; bf16-rounded float32."""
        wl, g = self.wl, self.wl.geom
        T = wl.T if T is None else T
        d, w = g.head_dim, wl.window
        K = np.empty((self.units, T, d), np.float32)
        V = np.empty((self.units, T, d), np.float32)
        Q = np.empty((self.units, g.group, w, d), np.float32)
        for u in range(self.units):
            K[u] = self._keys(u, T, record=True)
            V[u] = self.rng.standard_normal((T, d))
            Q[u] = self._queries(K[u], self._query_pool(u, T), g.group * w).reshape(g.group, w, d)
        shp = (g.batch, g.n_kv_heads)
        self._K = K
        return (bf16_round(K).reshape(*shp, T, d), bf16_round(V).reshape(*shp, T, d),
                bf16_round(Q).reshape(*shp, g.group, w, d))

    def decode(self, steps=None):
        """Per-step q [steps, b, Hq, d] and new k, v [steps, b, Hkv, d] (bf16-rounded).

        Decode queries follow the window-query recipe over the prefill keys."""
        wl, g = self.wl, self.wl.geom
        steps = wl.decode_steps if steps is None else steps
        d = g.head_dim
        q = np.empty((steps, self.units, g.group, d), np.float32)
        kn = np.empty((steps, self.units, d), np.float32)
        vn = np.empty((steps, self.units, d), np.float32)
        for u in range(self.units):
            Ku = self._K[u]
            q[:, u] = self._queries(Ku, self._query_pool(u, Ku.shape[0]), steps * g.group
                                    ).reshape(steps, g.group, d)
            if "scale" in self._params[u]:
                kn[:, u] = self.rng.standard_normal((steps, d)) * self._params[u]["scale"]
            else:
                comp = self.rng.integers(0, 16, steps)
                kn[:, u] = self._params[u]["means"][comp] + 0.5 * self.rng.standard_normal((steps, d))
            vn[:, u] = self.rng.standard_normal((steps, d))
        b, H = g.batch, g.n_kv_heads
        return (bf16_round(q).reshape(steps, b, H * g.group, d),
                bf16_round(kn).reshape(steps, b, H, d), bf16_round(vn).reshape(steps, b, H, d))


class TorchGenerator:
    """The same recipes as Generator, drawn with torch's generator on any
    device.  A multi-layer workload's prompts (about 19 GB at 36 layers of
    batch 4 x 32K) take minutes to draw with numpy on the host; on the GPU
    they take seconds.  The random streams differ from Generator's (and
    between devices), the distributions are the same.  Tensors come back as
    bf16 on `device`.  One generator per (seed, layer)."""

    def __init__(self, wl: Workload, seed: int = 0, layer: int = 0, device="cpu"):
        self.wl = wl
        self.dev = torch.device(device)
        self.gen = torch.Generator(device=self.dev)
        self.gen.manual_seed(int(seed) * 1000003 + int(layer) * 7919 + 17)
        g = wl.geom
        self.units = g.batch * g.n_kv_heads
        d = g.head_dim
        if wl.key_dist == "outlier":
            scale = torch.ones(self.units, d, device=self.dev)
            idx = torch.argsort(self._rand(self.units, d), dim=1)[:, :4]
            self.scale = scale.scatter_(1, idx, 6.0)
        elif wl.key_dist == "logscale":
            lo, hi = np.log(0.5), np.log(4.0)
            self.scale = torch.exp(lo + (hi - lo) * self._rand(self.units, d))
        elif wl.key_dist == "mixture":
            A = self._randn(self.units, d, 16).double()
            Qm, _ = torch.linalg.qr(A.cpu())                   # orthonormal columns, [units, d, 16]
            self.means = (Qm.transpose(1, 2) * np.sqrt(d)).float().to(self.dev)   # [units, 16, d]
            self.hot_comps = torch.argsort(self._rand(self.units, 16), dim=1)[:, :2]
        else:
            raise ValueError(wl.key_dist)
        self.scale = getattr(self, "scale", None)
        self._K = None
        self._pool = None

    def _rand(self, *shape):
        return torch.rand(*shape, generator=self.gen, device=self.dev)

    def _randn(self, *shape):
        return torch.randn(*shape, generator=self.gen, device=self.dev)

    def _randint(self, hi, shape):
        return torch.randint(0, hi, shape, generator=self.gen, device=self.dev)

    def _keys(self, n):
        d = self.wl.geom.head_dim
        if self.scale is not None:
            return self._randn(self.units, n, d) * self.scale[:, None, :], None
        comp = self._randint(16, (self.units, n))
        u = torch.arange(self.units, device=self.dev)[:, None]
        return self.means[u, comp] + 0.5 * self._randn(self.units, n, d), comp

    def _pools(self, comp, T):
        """Per unit, the candidate rows of the query recipe (None: all rows)."""
        if self.wl.key_dist == "outlier":
            return None
        if self.wl.key_dist == "logscale":
            n = max(3, T // 20)
            return [torch.sort(torch.argsort(self._rand(T), dim=0)[:n]).values for _ in range(self.units)]
        return [torch.nonzero(torch.isin(comp[u], self.hot_comps[u]))[:, 0] for u in range(self.units)]

    def _queries(self, n):
        """n queries per unit from its pool over the prefill keys: [units, n, d] float32."""
        K, pool = self._K, self._pool
        d = K.shape[-1]
        out = torch.empty(self.units, n, d, device=self.dev)
        for u in range(self.units):
            if pool is None:
                rows = self._randint(K.shape[1], (n, 3))
            else:
                rows = pool[u][self._randint(len(pool[u]), (n, 3))]
            v = K[u][rows].float().sum(dim=1)
            v = np.sqrt(d) * v / torch.linalg.norm(v, dim=1, keepdim=True)
            out[u] = v + 0.3 * self._randn(n, d)
        return out

    def prefill(self, T=None):
        """K, V [b, Hkv, T, d] and Q_obs [b, Hkv, g, w, d], bf16 on the device."""
        wl, g = self.wl, self.wl.geom
        T = wl.T if T is None else T
        d, w = g.head_dim, wl.window
        K, comp = self._keys(T)
        K = K.to(torch.bfloat16)
        V = self._randn(self.units, T, d).to(torch.bfloat16)
        self._K = K
        self._pool = self._pools(comp, T)
        Q = self._queries(g.group * w).to(torch.bfloat16)
        shp = (g.batch, g.n_kv_heads)
        return K.view(*shp, T, d), V.view(*shp, T, d), Q.view(*shp, g.group, w, d)

    def decode(self, steps=None):
        """q [steps, b, Hq, d], k_new, v_new [steps, b, Hkv, d], bf16 on the device;
        queries follow the window-query recipe over the prefill keys."""
        wl, g = self.wl, self.wl.geom
        steps = wl.decode_steps if steps is None else steps
        d = g.head_dim
        q = self._queries(steps * g.group).view(self.units, steps, g.group, d)
        kn, _ = self._keys(steps)
        vn = self._randn(self.units, steps, d)
        b, H = g.batch, g.n_kv_heads
        q = q.permute(1, 0, 2, 3).reshape(steps, b, H * g.group, d)
        kn = kn.permute(1, 0, 2).reshape(steps, b, H, d)
        vn = vn.permute(1, 0, 2).reshape(steps, b, H, d)
        return q.to(torch.bfloat16), kn.to(torch.bfloat16), vn.to(torch.bfloat16)


def random_moments(rng, batch, n_kv_heads, d, n=4096, scale=0.05):
    """Fixed dense moments (n, mu_k, mu_v, C) for decode-only workloads."""
    shp = (batch, n_kv_heads)
    return (np.full(shp, n, np.int32),
            (scale * rng.standard_normal((*shp, d))).astype(np.float32),
            (scale * rng.standard_normal((*shp, d))).astype(np.float32),
            (scale * rng.standard_normal((*shp, d, d))).astype(np.float32))


def random_cache(rng, batch, n_kv_heads, d, length, key_scale=1.0):
    """A retained cache of `length` rows per unit: N(0,1) keys/values (bf16-rounded)."""
    shp = (batch, n_kv_heads, length, d)
    return (bf16_round(key_scale * rng.standard_normal(shp)),
            bf16_round(rng.standard_normal(shp)))


def random_queries(rng, batch, n_q_heads, d, norm=None):
    """Decode queries; if `norm` is given each row is rescaled to that norm."""
    q = rng.standard_normal((batch, n_q_heads, d))
    if norm is not None:
        q = norm * q / np.linalg.norm(q, axis=-1, keepdims=True)
    return bf16_round(q)
