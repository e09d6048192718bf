"""The near-tie parity helpers the GPU tests use (tests/parity.py), on the
CPU against the oracle itself: following the oracle's own evictions
reproduces its result, a row the oracle would not evict is rejected, an exact
tie accepts either row, and the compress checker accepts the oracle's own
result and rejects a swapped row."""
import numpy as np
import pytest

import oracle as O
from paper_2606_01563_gb300.inputs import bf16_round
from parity import check_compress_unit, evict_scores, follow_evictions, near_minimal


def _state(rng, L, d, n_e, G=2):
    K = bf16_round(1.5 * rng.standard_normal((L, d)))
    V = bf16_round(rng.standard_normal((L, d)))
    q = bf16_round(2.0 * rng.standard_normal((G, d)))
    m = O.moments_of(bf16_round(rng.standard_normal((n_e, d))), bf16_round(rng.standard_normal((n_e, d))))
    return q, K, V, np.arange(L) * 3, m


def test_follow_reproduces_the_oracle():
    rng = np.random.default_rng(1)
    q, K, V, pos, m = _state(rng, 40, 32, 50)
    r = O.evict_append(q, K, V, pos, m, 25, 1e-6)
    assert min(r.gaps) > 1e-5
    f = follow_evictions(q, K, V, pos, m, 25, 1e-6, r.evicted_pos)
    np.testing.assert_array_equal(f.pos, r.pos)
    np.testing.assert_array_equal(f.K, r.K)
    assert f.moments.n == r.moments.n and f.ties == 0
    np.testing.assert_allclose(f.moments.C, r.moments.C, atol=1e-12)
    np.testing.assert_allclose(f.moments.mu_k, r.moments.mu_k, atol=1e-12)
    # the first step's scores: the oracle's first eviction is their strict argmin
    sc = evict_scores(q, K, V, m, 1e-6)
    assert near_minimal(sc) == [int(np.argmin(sc))] and pos[np.argmin(sc)] == r.evicted_pos[0]


def test_follow_rejects_a_row_the_oracle_keeps():
    rng = np.random.default_rng(2)
    q, K, V, pos, m = _state(rng, 30, 32, 0)
    r = O.evict_append(q, K, V, pos, m, 20, 0.0)
    kept_pos = [p for p in pos if p not in r.evicted_pos]
    wrong = list(r.evicted_pos[:-1]) + [kept_pos[0]]
    with pytest.raises(AssertionError):
        follow_evictions(q, K, V, pos, m, 20, 0.0, wrong)


def test_follow_accepts_either_row_of_an_exact_tie():
    rng = np.random.default_rng(3)
    q, K, V, pos, m = _state(rng, 12, 16, 0, G=1)
    sc = evict_scores(q, K, V, m, 0.0)
    j = int(np.argmin(sc))
    # a second copy of the minimal row at the end: the two tie exactly
    K2, V2 = np.vstack([K, K[j:j + 1]]), np.vstack([V, V[j:j + 1]])
    pos2 = np.append(pos, 1000)
    r = O.evict_append(q, K2, V2, pos2, m, 12, 0.0)
    assert r.evicted_pos == [pos[j]]  # the oracle breaks the tie to the lower position
    for pick in (pos[j], 1000):
        f = follow_evictions(q, K2, V2, pos2, m, 12, 0.0, [pick])
        assert f.ties == 1 and pick not in f.pos


def _compress_out(ref, K, V, T, B):
    """A kernel's outputs as the oracle would write them (one unit)."""
    R = ref.idx
    s2 = np.where(np.isfinite(ref.score2), ref.score2, 0.0)
    return {"K": K[R][None, None], "V": V[R][None, None], "pos": np.asarray(R)[None, None],
            "len": np.array([[len(R)]]), "seen": np.array([[T]]), "n": np.array([[ref.moments.n]]),
            "mu_k": ref.moments.mu_k[None, None], "mu_v": ref.moments.mu_v[None, None],
            "C": ref.moments.C[None, None], "s": ref.scores[None, None], "s2": s2[None, None],
            "i1": np.asarray(ref.idx_stage1)[None, None]}


def test_compress_checker_accepts_the_oracle_and_rejects_a_swap():
    rng = np.random.default_rng(4)
    T, d, B, w = 300, 32, 40, 8
    K = bf16_round(rng.standard_normal((T, d)))
    V = bf16_round(rng.standard_normal((T, d)))
    Q = bf16_round(2.0 * rng.standard_normal((2, w, d)))
    ref = O.compress(K, V, Q, B, w, 1, True, 1, True, 1e-6)
    out = _compress_out(ref, K, V, T, B)
    assert check_compress_unit(out, 0, 0, K, V, Q, T, B, w, 1, True, 1, 1, 1e-6) == (ref.gap1 > 1e-5 and ref.gap2 > 1e-5)
    bad = dict(out)
    pos = out["pos"].copy()
    free = [t for t in range(1, T - w) if t not in set(ref.idx)]
    i = next(i for i, p in enumerate(pos[0, 0]) if 1 <= p < T - w)
    pos[0, 0, i] = free[0]
    bad["pos"] = np.sort(pos, axis=-1)
    with pytest.raises(AssertionError):
        check_compress_unit(bad, 0, 0, K, V, Q, T, B, w, 1, True, 1, 1, 1e-6)
