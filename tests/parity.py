"""Parity checks of the GPU selections against the fp64 oracle that hold at
near ties.

The oracle decides a selection exactly only where its boundary (or argmin)
gap exceeds GAP_EXACT (relative).  Below that gap either side of the
boundary is a correct answer, so these helpers check what is unique and
that the rest is valid:
  - compress: each selection is replayed on the kernel's own fp32 scores
    (the radix select must return exactly the top k of the values it
    ranked, lower position first on ties); where the oracle's gap exceeds
    GAP_EXACT it must also equal the oracle's set; otherwise the oracle
    continues from the kernel's choice (score2 under the kernel's stage-1
    set, moments of the kernel's evicted set), so scores, rows and moments
    are still compared element by element;
  - eviction (Algorithm 1 Phase 1): the kernel reports only the surviving
    rows, so the oracle follows it: at every step it recomputes the scores
    of Algorithm 1 (alpha_j ||r_j||, from the oracle's own functions) under
    the state reached so far, and the evicted row must be the argmin, or,
    at a near tie, one of the near-minimal rows that the kernel evicted
    (a depth-first search over those, which are rare); the state then
    follows that row.  The surviving rows and the moments reached are then
    compared with the kernel's.
"""
import numpy as np

import oracle as O
from gpu_util import GAP_EXACT, assert_moment_close


# ----------------------------------------------------------------- compress
def score2_under(K, V, s, R0, tau):
    """Oracle score2 (Eq. residual under the moments of all \\ R0, times s) for a
    given stage-1 set R0 (protected rows included)."""
    keep0 = np.zeros(K.shape[0], bool)
    keep0[R0] = True
    r = O.residual(K, V, O.moments_of(K[~keep0], V[~keep0]), tau)
    return s * np.sqrt((r * r).sum(axis=1))


def evicted_moments(K, V, R):
    keep = np.zeros(K.shape[0], bool)
    keep[R] = True
    return O.moments_of(K[~keep], V[~keep])


def check_rows_and_moments(out, bi, h, K, V, R, m):
    n_r = len(R)
    np.testing.assert_array_equal(out["K"][bi, h, :n_r], K[R])
    np.testing.assert_array_equal(out["V"][bi, h, :n_r], V[R])
    assert out["n"][bi, h] == m.n
    if m.n:
        assert_moment_close(out["mu_k"][bi, h], m.mu_k, "mu_k")
        assert_moment_close(out["mu_v"][bi, h], m.mu_v, "mu_v")
        assert_moment_close(out["C"][bi, h], m.C, "C")
    else:
        assert not out["C"][bi, h].any()


def check_compress_unit(out, bi, h, K, V, Q, T, B, window, sink, keep_window, pool, mi, tau):
    """One (batch, KV head) unit of a per-unit-budget mkv_compress.

    out: host copies of the cache ("K", "V", "pos", "len", "seen"), moments
    ("n", "mu_k", "mu_v", "C") and the diagnostics ("s", "s2", "i1").
    Returns True when every selection was decided exactly by the oracle."""
    ref = O.compress(K, V, Q, B, window, sink, keep_window, pool, bool(mi), tau)
    s_g = np.asarray(out["s"][bi, h], np.float64)
    np.testing.assert_allclose(s_g, ref.scores, rtol=2e-5, atol=2e-6 * ref.scores.max())
    assert out["seen"][bi, h] == T
    if T <= B:
        assert out["len"][bi, h] == T
        np.testing.assert_array_equal(out["pos"][bi, h, :T], np.arange(T))
        check_rows_and_moments(out, bi, h, K, V, np.arange(T), O.Moments.zeros(K.shape[1]))
        return True
    prot = O.protected_mask(T, window, sink, keep_window)
    free = ~prot
    k = B - int(prot.sum())
    # stage 1: the kernel's choice is the exact top k of its own scores
    R0 = out["i1"][bi, h]
    np.testing.assert_array_equal(R0, O.select_topk(s_g, k, prot)[0])
    exact1 = ref.gap1 > GAP_EXACT
    if exact1:
        np.testing.assert_array_equal(R0, ref.idx_stage1)
    assert out["len"][bi, h] == B
    R = out["pos"][bi, h, :B]
    if mi:
        s2_g = np.asarray(out["s2"][bi, h], np.float64)
        score2 = ref.score2 if exact1 else score2_under(K, V, ref.scores, R0, tau)
        np.testing.assert_allclose(s2_g[free], score2[free], rtol=1e-4, atol=1e-5 * score2[free].max())
        np.testing.assert_array_equal(R, O.select_topk(s2_g, k, prot)[0])
        exact = exact1 and ref.gap2 > GAP_EXACT
    else:
        np.testing.assert_array_equal(R, R0)
        exact = exact1
    if exact:
        np.testing.assert_array_equal(R, ref.idx)
        m = ref.moments
    else:
        m = evicted_moments(K, V, R)
    check_rows_and_moments(out, bi, h, K, V, R, m)
    return exact


def check_compress_item_adaptive(out, bi, K, V, Q, T, B, window, sink, keep_window, pool, mi, tau):
    """The KV heads of batch item bi with the budget shared across them
    (K, V: [H, T, d]); out as for check_compress_unit, "i1" [b, H*B] of h*T+t."""
    H = K.shape[0]
    ref = O.compress_adaptive(K, V, Q, B, window, sink, keep_window, pool, bool(mi), tau)
    s_g = np.asarray(out["s"][bi], np.float64)
    for h in range(H):
        np.testing.assert_allclose(s_g[h], ref.scores[h], rtol=2e-5, atol=2e-6 * ref.scores[h].max())
    assert (out["seen"][bi] == T).all()
    if T <= B:
        for h in range(H):
            assert out["len"][bi, h] == T
            np.testing.assert_array_equal(out["pos"][bi, h, :T], np.arange(T))
            assert out["n"][bi, h] == 0
        return True
    prot = np.stack([O.protected_mask(T, window, sink, keep_window)] * H)
    k = H * B - int(prot.sum())

    def flat(lists):
        return np.concatenate([h * T + np.asarray(r) for h, r in enumerate(lists)])

    R0 = O.select_topk_joint(s_g, k, prot)[0]
    np.testing.assert_array_equal(out["i1"][bi], flat(R0))
    exact1 = ref.gap1 > GAP_EXACT
    if exact1:
        np.testing.assert_array_equal(flat(R0), flat(ref.idx_stage1))
    assert out["len"][bi].sum() == H * B
    R = [out["pos"][bi, h, :out["len"][bi, h]] for h in range(H)]
    if mi:
        s2_g = np.asarray(out["s2"][bi], np.float64)
        score2 = ref.score2 if exact1 else np.stack([score2_under(K[h], V[h], ref.scores[h], R0[h], tau)
                                                     for h in range(H)])
        for h in range(H):
            free = ~prot[h]
            np.testing.assert_allclose(s2_g[h][free], score2[h][free], rtol=1e-4,
                                       atol=1e-5 * score2[h][free].max())
        np.testing.assert_array_equal(flat(R), flat(O.select_topk_joint(s2_g, k, prot)[0]))
        exact = exact1 and ref.gap2 > GAP_EXACT
    else:
        np.testing.assert_array_equal(flat(R), flat(R0))
        exact = exact1
    if exact:
        np.testing.assert_array_equal(flat(R), flat(ref.idx))
    for h in range(H):
        m = ref.moments[h] if exact else evicted_moments(K[h], V[h], R[h])
        check_rows_and_moments(out, bi, h, K[h], V[h], R[h], m)
    return exact


# ------------------------------------------------------------------ eviction
def evict_scores(q, K, V, m, tau):
    """The scores of one step of Algorithm 1 Phase 1 under moments m:
    alpha_j ||r_j|| with alpha summed over the group's query heads and r_j
    the moment residual (Eq. residual; r_j = v_j with no evicted token)."""
    alpha = O.group_attention_weights(q, K)
    r = O.residual(K, V, m, tau)
    return alpha * np.sqrt((r * r).sum(axis=1))


def near_minimal(scores):
    """Rows whose score is within GAP_EXACT (relative, as the oracle measures
    its argmin gap) of the smallest, lowest row first."""
    s_min = scores.min()
    return [j for j in range(len(scores)) if scores[j] - s_min <= GAP_EXACT * abs(scores[j])]


class EvictFollow:
    """The oracle's state after following the kernel's evictions."""

    def __init__(self, K, V, pos, m, ties):
        self.K, self.V, self.pos, self.moments, self.ties = K, V, pos, m, ties


def follow_evictions(q, K, V, pos, m, budget, tau, evicted_by_kernel):
    """Algorithm 1 Phase 1 on (K, V, pos, m) down to `budget` rows, each step
    taking the oracle's argmin, or at a near tie one of the near-minimal rows
    in `evicted_by_kernel` (positions); fails if the kernel evicted a row the
    oracle never could.  The raw sums follow Eq. app_update (oracle
    add_token_sums).  Returns an EvictFollow."""
    want = set(int(p) for p in evicted_by_kernel)
    K = np.asarray(K, np.float64)
    V = np.asarray(V, np.float64)
    pos = np.asarray(pos, np.int64)
    assert len(want) == max(0, len(pos) - budget), (len(want), len(pos), budget)

    def go(K, V, pos, sums, left, ties):
        if len(pos) <= budget:
            assert not left, f"kernel evicted {sorted(left)} beyond the oracle's path"
            return EvictFollow(K, V, pos, O.from_sums(*sums), ties)
        sc = evict_scores(q, K, V, O.from_sums(*sums), tau)
        cands = near_minimal(sc)
        allowed = [j for j in cands if int(pos[j]) in left]
        assert allowed, (f"kernel kept every near-minimal row {[int(pos[j]) for j in cands]} "
                         f"(scores {sc[cands]}, min {sc.min()})")
        err = None
        for j in allowed:
            keep = np.ones(len(pos), bool)
            keep[j] = False
            try:
                return go(K[keep], V[keep], pos[keep], O.add_token_sums(sums, K[j], V[j]),
                          left - {int(pos[j])}, ties + (len(cands) > 1))
            except AssertionError as e:  # that branch of a near tie does not lead to the kernel's set
                err = e
        raise err

    return go(K, V, pos, O.to_sums(m), want, 0)


def check_evicted_unit(gpu, bi, h, q, K, V, pos, m, budget, tau):
    """Checks one unit of an mkv_evict_append result (host copies in `gpu`)
    against the oracle following the kernel's evictions; returns the
    EvictFollow state."""
    L = int(gpu["len"][bi, h])
    kept = gpu["pos"][bi, h, :L]
    assert np.all(np.diff(kept) > 0), "surviving rows out of position order"
    assert set(kept.tolist()) <= set(np.asarray(pos).tolist())
    evicted = sorted(set(np.asarray(pos).tolist()) - set(kept.tolist()))
    f = follow_evictions(q, K, V, pos, m, budget, tau, evicted)
    np.testing.assert_array_equal(kept, f.pos)
    if L:
        np.testing.assert_array_equal(gpu["K"][bi, h, :L], f.K)
        np.testing.assert_array_equal(gpu["V"][bi, h, :L], f.V)
    assert gpu["n"][bi, h] == f.moments.n
    if f.moments.n:
        assert_moment_close(gpu["mu_k"][bi, h], f.moments.mu_k, "mu_k")
        assert_moment_close(gpu["mu_v"][bi, h], f.moments.mu_v, "mu_v")
        assert_moment_close(gpu["C"][bi, h], f.moments.C, "C")
    return f
