"""Pins for the fp64 oracle: each test checks the oracle against something the
paper or mathematics fixes independently of the oracle's own formulas --
library attention (torch SDPA in float64), the Taylor expansion measured by
finite differences, identities and bounds printed in the paper, exhaustive
search on tiny inputs, and Table 5's storage figures.
"""
import itertools
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch
import torch.nn.functional as F
from scipy.special import logsumexp

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# --------------------------------------------------------------------------
# independent brute-force helpers (library attention, finite differences)
# --------------------------------------------------------------------------

def sdpa(q, K, V, mask=None):
    """Library attention in float64: q [n_q, d] or [d]."""
    q = np.atleast_2d(np.asarray(q, np.float64))
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a, np.float64))[None, None]
    m = None if mask is None else torch.from_numpy(mask)
    o = F.scaled_dot_product_attention(t(q), t(K), t(V), attn_mask=m)
    return o[0, 0].numpy()


def attn_weights(q, K, mask=None):
    """Softmax weights via library attention over one-hot values."""
    K = np.asarray(K, np.float64)
    return sdpa(q, K, np.eye(K.shape[0]), mask)


def brute_logZ(q, K):
    K = np.asarray(K, np.float64)
    return float(torch.logsumexp(torch.from_numpy(K @ np.asarray(q, np.float64) / math.sqrt(K.shape[1])), 0))


def fd_jacobian_at_zero(K_E, V_E, h=1e-4):
    """Central-difference Jacobian of f_E(q) at q = 0 (library attention)."""
    d = K_E.shape[1]
    J = np.zeros((V_E.shape[1], d))
    for b in range(d):
        e = np.zeros(d)
        e[b] = h
        J[:, b] = (sdpa(e, K_E, V_E)[0] - sdpa(-e, K_E, V_E)[0]) / (2 * h)
    return J


def rng(seed=0):
    return np.random.default_rng(seed)


# --------------------------------------------------------------------------
# Sec. 2: attention and its decomposition
# --------------------------------------------------------------------------

def test_full_attention_matches_library():
    r = rng(1)
    K, V, q = r.standard_normal((37, 16)), r.standard_normal((37, 16)), 2 * r.standard_normal(16)
    f, lz = O.full_attention(q, K, V)
    np.testing.assert_allclose(f, sdpa(q, K, V)[0], rtol=0, atol=1e-13)
    assert abs(lz - brute_logZ(q, K)) < 1e-12


def test_decomposition_is_exact():
    """Eq. decomposition: f = w_R f_R + w_E f_E with w = Z_part / Z."""
    r = rng(2)
    K, V, q = r.standard_normal((40, 8)), r.standard_normal((40, 8)), r.standard_normal(8)
    keep = r.random(40) < 0.4
    f_R, lR, f_E, lE = O.sub_outputs(q, K, V, keep)
    lZ = logsumexp([lR, lE])
    f = math.exp(lR - lZ) * f_R + math.exp(lE - lZ) * f_E
    np.testing.assert_allclose(f, sdpa(q, K, V)[0], atol=1e-13)
    np.testing.assert_allclose(f_R, sdpa(q, K[keep], V[keep])[0], atol=1e-13)


# --------------------------------------------------------------------------
# Sec. 4.1 / App. A.1: moments
# --------------------------------------------------------------------------

def test_s_tilde_identity_exact_rationals():
    """S_tilde from the definition equals S - s_v s_k^T / n (Eq. app_S_tilde),
    checked against exact rational arithmetic on a small integer set."""
    K = [[1, -2, 3], [0, 4, -1], [2, 2, 2], [-3, 1, 0]]
    V = [[2, 0, -1], [1, 1, 1], [-2, 3, 0], [0, -1, 5]]
    n = len(K)
    s_k = [sum(Fraction(k[b]) for k in K) for b in range(3)]
    s_v = [sum(Fraction(v[a]) for v in V) for a in range(3)]
    S = [[sum(Fraction(v[a] * k[b]) for k, v in zip(K, V)) for b in range(3)] for a in range(3)]
    S_tilde = [[S[a][b] - s_v[a] * s_k[b] / n for b in range(3)] for a in range(3)]
    m = O.moments_of(np.array(K, float), np.array(V, float))
    assert m.n == 4
    np.testing.assert_allclose(m.mu_k, [float(x / n) for x in s_k], atol=1e-15)
    np.testing.assert_allclose(m.mu_v, [float(x / n) for x in s_v], atol=1e-15)
    np.testing.assert_allclose(m.C, [[float(x / n) for x in row] for row in S_tilde], atol=1e-14)


def test_incremental_equals_batch():
    """Raw-sum updates (Eq. app_update), the Welford form and Chan merges all
    reproduce the batch moments of the same set."""
    r = rng(3)
    d, n = 12, 57
    K = 3 * r.standard_normal((n, d)) + 5.0
    V = r.standard_normal((n, d)) - 2.0
    batch = O.moments_of(K, V)
    sums = (0, np.zeros(d), np.zeros(d), np.zeros((d, d)))
    wel = O.Moments.zeros(d)
    for i in range(n):
        sums = O.add_token_sums(sums, K[i], V[i])
        wel = O.add_token_welford(wel, K[i], V[i])
    via_sums = O.from_sums(*sums)
    cuts = [0, 5, 6, 30, n]
    parts = [O.moments_of(K[a:b], V[a:b]) for a, b in zip(cuts[:-1], cuts[1:])]
    merged = parts[0]
    for p in parts[1:]:
        merged = O.merge_chan(merged, p)
    for m in (via_sums, wel, merged):
        assert m.n == n
        np.testing.assert_allclose(m.mu_k, batch.mu_k, atol=1e-12)
        np.testing.assert_allclose(m.mu_v, batch.mu_v, atol=1e-12)
        np.testing.assert_allclose(m.C, batch.C, atol=1e-12)
    # round trip through the raw sums
    back = O.from_sums(*O.to_sums(batch))
    np.testing.assert_allclose(back.C, batch.C, atol=1e-12)


def test_zero_sum_of_centered_logits():
    """sum_i delta_i = 0 for any query (Eq. app_zero_sum)."""
    r = rng(4)
    K = r.standard_normal((31, 16)) * 3
    for _ in range(5):
        assert abs(O.centered_logits(r.standard_normal(16) * 4, K).sum()) < 1e-11


# --------------------------------------------------------------------------
# Eq. fhat is the first-order expansion of f_E; Eq. residual uses it
# --------------------------------------------------------------------------

def test_fhat_is_first_order_taylor_of_fE():
    """f_hat_E(q) = f_E(0) + J q with J the Jacobian of library attention at
    q = 0 (the expansion exp(delta) ~ 1 + delta of Sec. 4.1), and the gap to
    the exact f_E shrinks quadratically (App. A.2)."""
    r = rng(5)
    d, n = 8, 20
    K_E = r.standard_normal((n, d))
    V_E = r.standard_normal((n, d)) + np.arange(d)  # non-symmetric structure
    m = O.moments_of(K_E, V_E)
    f0 = sdpa(np.zeros(d), K_E, V_E)[0]
    J = fd_jacobian_at_zero(K_E, V_E)
    for _ in range(3):
        q = r.standard_normal(d)
        np.testing.assert_allclose(O.fhat_E(q, m), f0 + J @ q, atol=1e-7)
    q = r.standard_normal(d)
    errs = [np.linalg.norm(sdpa(e * q, K_E, V_E)[0] - O.fhat_E(e * q, m)) for e in (0.02, 0.01)]
    assert 3.6 < errs[0] / errs[1] < 4.4
    np.testing.assert_allclose(O.fhat_E(q, m, order=0), V_E.mean(axis=0), atol=1e-14)


def test_residual_is_value_minus_affine_model():
    """r_j = v_j - (f_E(0) + J k_j): the residual is each value minus the
    first-order model of the evicted output evaluated at its own key."""
    r = rng(6)
    d = 6
    K_E, V_E = r.standard_normal((15, d)), r.standard_normal((15, d)) * 2 + 1
    K, V = r.standard_normal((9, d)), r.standard_normal((9, d))
    m = O.moments_of(K_E, V_E)
    f0 = sdpa(np.zeros(d), K_E, V_E)[0]
    J = fd_jacobian_at_zero(K_E, V_E)
    np.testing.assert_allclose(O.residual(K, V, m), V - f0 - K @ J.T, atol=1e-7)
    np.testing.assert_allclose(O.residual(K, V, O.Moments.zeros(d)), V, atol=0)


# --------------------------------------------------------------------------
# App. B: Jensen estimate, tightness, mixing weight
# --------------------------------------------------------------------------

def test_jensen_lower_bound_and_tightness():
    r = rng(7)
    d, n = 16, 40
    c = r.standard_normal(d) * 2
    D = r.standard_normal((n, d))
    q = r.standard_normal(d) * 2
    prev = None
    for eps in (0.08, 0.04, 0.02):
        K_E = c + eps * D
        m = O.moments_of(K_E, np.zeros((n, d)))
        lz, lzh = brute_logZ(q, K_E), O.log_zhat_E(q, m)
        assert lzh <= lz + 1e-14                       # Eq. jensen
        Sigma = np.cov(K_E.T, bias=True)
        var = q @ Sigma @ q / d                          # Eq. app_logit_var
        assert abs(var - np.mean(O.centered_logits(q, K_E) ** 2)) < 1e-12
        resid = math.exp(lz - lzh) - 1 - 0.5 * var       # Eq. app_ratio remainder
        if prev is not None:
            assert abs(resid) < abs(prev) / 6            # O(sigma^3): x8 per halving
        prev = resid


def test_weight_bias_identity():
    """Eq. app_weight_bias.  Its middle line, Z_R eps Z_hat_E /
    ((Z_R + Z_hat_E)(Z_R + Z_E)), equals w_R w_hat_E eps and also
    w_hat_R w_hat_E eps / (1 + eps w_hat_E); the printed last form, with w_R
    and the denominator together, is not equal to it (reading: a typo for
    w_hat_R), so both consistent forms are checked."""
    r = rng(8)
    d = 16
    K, V = r.standard_normal((50, d)), r.standard_normal((50, d))
    keep = np.arange(50) < 20
    q = r.standard_normal(d) * 2
    m = O.moments_of(K[~keep], V[~keep])
    out, lse = O.corrected_output(q, K[keep], V[keep], m)
    lR, lE = brute_logZ(q, K[keep]), brute_logZ(q, K[~keep])
    w_hat_R = math.exp(lR - lse)
    w_R = math.exp(lR - logsumexp([lR, lE]))
    lEh = O.log_zhat_E(q, m)
    eps = math.exp(lE - lEh) - 1
    w_hat_E = 1 - w_hat_R
    mid = math.exp(lR) * eps * math.exp(lEh) / (
        (math.exp(lR) + math.exp(lEh)) * (math.exp(lR) + math.exp(lE)))
    assert abs((w_hat_R - w_R) - mid) < 1e-12
    assert abs((w_hat_R - w_R) - w_R * w_hat_E * eps) < 1e-12
    assert abs((w_hat_R - w_R) - w_hat_R * w_hat_E * eps / (1 + eps * w_hat_E)) < 1e-12
    # the output is the Eq. fused mixture of library f_R and f_hat_E
    np.testing.assert_allclose(out, w_hat_R * sdpa(q, K[keep], V[keep])[0]
                               + w_hat_E * O.fhat_E(q, m), atol=1e-12)


# --------------------------------------------------------------------------
# Phase 2 special cases (Algorithm 1)
# --------------------------------------------------------------------------

def test_no_evicted_tokens_gives_plain_attention():
    r = rng(9)
    K, V, q = r.standard_normal((33, 16)), r.standard_normal((33, 16)), r.standard_normal((4, 16))
    out, lse, _, _ = O.decode_step(q, K, V, O.Moments.zeros(16))
    np.testing.assert_allclose(out, sdpa(q, K, V), atol=1e-13)
    np.testing.assert_allclose(lse, logsumexp(q @ K.T / 4.0, axis=1), atol=1e-12)
    # append first (Algorithm 1 adds the new token to R before attending)
    kn, vn = r.standard_normal(16), r.standard_normal(16)
    out2, _, K2, _ = O.decode_step(q, K, V, O.Moments.zeros(16), kn, vn)
    assert K2.shape[0] == 34
    np.testing.assert_allclose(out2, sdpa(q, np.vstack([K, kn]), np.vstack([V, vn])), atol=1e-13)
    # correction switched off ignores the moments
    m = O.moments_of(r.standard_normal((5, 16)), r.standard_normal((5, 16)))
    out3, _, _, _ = O.decode_step(q, K, V, m, correction=False)
    np.testing.assert_allclose(out3, sdpa(q, K, V), atol=1e-13)


def test_single_evicted_token_is_exact():
    """n_e = 1: delta = 0, S_tilde = 0, Z_hat_E = Z_E, so the corrected output
    is full attention over R and the evicted token exactly."""
    r = rng(10)
    d = 16
    K, V = r.standard_normal((21, d)), r.standard_normal((21, d))
    q = r.standard_normal((3, d)) * 2
    m = O.moments_of(K[20:], V[20:])
    out, lse, _, _ = O.decode_step(q, K[:20], V[:20], m)
    np.testing.assert_allclose(out, sdpa(q, K, V), atol=1e-13)
    np.testing.assert_allclose(lse, logsumexp(q @ K.T / 4.0, axis=1), atol=1e-12)


def test_identical_evicted_keys_are_exact():
    r = rng(11)
    d = 8
    K, V = r.standard_normal((30, d)), r.standard_normal((30, d))
    K[10:] = K[10]
    m = O.moments_of(K[10:], V[10:])
    q = r.standard_normal((2, d))
    out, _, _, _ = O.decode_step(q, K[:10], V[:10], m)
    np.testing.assert_allclose(out, sdpa(q, K, V), atol=1e-12)


def test_empty_retained_set_uses_moment_term():
    r = rng(12)
    d = 8
    K_E, V_E = r.standard_normal((9, d)), r.standard_normal((9, d))
    m = O.moments_of(K_E, V_E)
    q = r.standard_normal(d)
    out, lse = O.corrected_output(q, np.zeros((0, d)), np.zeros((0, d)), m)
    np.testing.assert_allclose(out, O.fhat_E(q, m))
    assert abs(lse - (math.log(9) + q @ K_E.mean(0) / math.sqrt(d))) < 1e-12
    with pytest.raises(ValueError):
        O.corrected_output(q, np.zeros((0, d)), np.zeros((0, d)), O.Moments.zeros(d))


def test_error_bound_and_second_order_convergence():
    """||f_E - f_hat_E|| stays under the leading term of Eq. app_error_bound and
    shrinks as the square of the evicted key spread."""
    r = rng(13)
    d, n = 16, 64
    c, D = r.standard_normal(d), r.standard_normal((n, d))
    V_E = r.standard_normal((n, d))
    q = r.standard_normal(d) * 2
    errs = []
    for eps in (0.4, 0.2, 0.1, 0.05):
        K_E = c + eps * D
        err = np.linalg.norm(sdpa(q, K_E, V_E)[0] - O.fhat_E(q, O.moments_of(K_E, V_E)))
        bound, sigma = O.error_bound(q, K_E, V_E)
        assert err <= bound * (1 + sigma)   # leading term; O(sigma^4) slack
        errs.append(err)
    slopes = [math.log2(a / b) for a, b in zip(errs[:-1], errs[1:])]
    assert all(1.8 < s < 2.2 for s in slopes[1:]), slopes


def test_self_regulation_limits():
    """App. B.2: as sigma -> 0 the corrected output tends to f; as sigma grows
    the estimated evicted weight w_hat_E goes to 0."""
    r = rng(14)
    d = 16
    K_R, V_R = r.standard_normal((20, d)), r.standard_normal((20, d))
    c, D, V_E = r.standard_normal(d), r.standard_normal((30, d)), r.standard_normal((30, d))
    q = r.standard_normal(d) * 2
    gaps = []
    for eps in (0.1, 0.01, 0.001):
        K_E = c + eps * D
        out, _ = O.corrected_output(q, K_R, V_R, O.moments_of(K_E, V_E))
        gaps.append(np.linalg.norm(out - sdpa(q, np.vstack([K_R, K_E]), np.vstack([V_R, V_E]))[0]))
    assert gaps[2] < gaps[1] < gaps[0] and gaps[2] < 1e-6
    # large spread at a fixed true evicted mass (the centroid slides along q so
    # that Z_E stays put): Z_hat_E / Z_E -> 0 and w_hat_E -> 0 (Eq. app_what_e)
    Dc = D - D.mean(axis=0)
    lZR = brute_logZ(q, K_R)
    ratios, w_hats, w_trues = [], [], []
    for eps in (1.0, 4.0, 16.0):
        lme = brute_logZ(q, eps * Dc) - math.log(len(Dc))
        K_E = c - lme * math.sqrt(d) * q / (q @ q) + eps * Dc
        m = O.moments_of(K_E, V_E)
        _, lse = O.corrected_output(q, K_R, V_R, m)
        w_hat_E = 1 - math.exp(lZR - lse)
        lZE = brute_logZ(q, K_E)
        w_E = math.exp(lZE - logsumexp([lZR, lZE]))
        w_R = math.exp(lZR - logsumexp([lZR, lZE]))
        ratio = math.exp(O.log_zhat_E(q, m) - lZE)
        assert abs(w_hat_E - w_E * ratio / (w_R + w_E * ratio)) < 1e-12
        ratios.append(ratio)
        w_hats.append(w_hat_E)
        w_trues.append(w_E)
    assert max(w_trues) - min(w_trues) < 1e-9
    assert ratios[0] > ratios[1] > ratios[2] and ratios[2] < 1e-6
    assert w_hats[0] > w_hats[1] > w_hats[2] and w_hats[2] < 1e-6


def test_constructed_near_orthogonal_case():
    """Retained values in span(e1..e8), evicted values in span(e9..e16),
    evicted keys clustered: the corrected output is closer to full attention
    than renormalised attention over R (the directional gap of Sec. 3)."""
    r = rng(15)
    d, L, n = 16, 32, 32
    K_R = r.standard_normal((L, d)) * 1.5
    V_R = np.zeros((L, d)); V_R[:, :8] = r.standard_normal((L, 8))
    c = r.standard_normal(d) * 1.5
    K_E = c + 0.05 * r.standard_normal((n, d))
    V_E = np.zeros((n, d)); V_E[:, 8:] = r.standard_normal((n, 8)) + 1.0
    m = O.moments_of(K_E, V_E)
    K, V = np.vstack([K_R, K_E]), np.vstack([V_R, V_E])
    for _ in range(8):
        q = r.standard_normal(d) * 2
        f = sdpa(q, K, V)[0]
        out, _ = O.corrected_output(q, K_R, V_R, m)
        assert np.linalg.norm(f - out) < np.linalg.norm(f - sdpa(q, K_R, V_R)[0])


# --------------------------------------------------------------------------
# Prefill pieces (Sec. 5.1)
# --------------------------------------------------------------------------

def test_window_scores_match_library_attention():
    r = rng(16)
    T, d, g, w = 50, 8, 2, 5
    K = r.standard_normal((T, d)) * 2
    Q = r.standard_normal((g, w, d)) * 2
    mask = np.zeros((w, T), bool)
    for i in range(w):
        mask[i, :T - w + i + 1] = True
    expect = sum(attn_weights(Q[h], K, mask).sum(axis=0) for h in range(g))
    np.testing.assert_allclose(O.window_scores(Q, K), expect, atol=1e-13)
    expect_nc = sum(attn_weights(Q[h], K).sum(axis=0) for h in range(g))
    np.testing.assert_allclose(O.window_scores(Q, K, causal=False), expect_nc, atol=1e-13)
    assert abs(O.window_scores(Q, K).sum() - g * w) < 1e-12


def test_pool_scores_aligned_chunks():
    np.testing.assert_allclose(O.pool_scores([1, 2, 3, 4, 5], 2), [3, 3, 7, 7, 5])
    np.testing.assert_allclose(O.pool_scores([1, 2, 3, 4, 5], 4), [10, 10, 10, 10, 5])
    np.testing.assert_allclose(O.pool_scores([1, 2, 3], 1), [1, 2, 3])


def test_select_topk_exhaustive():
    """The selected set is the unique k-subset whose every member precedes
    every rejected candidate in (higher score, lower position) order."""
    r = rng(17)
    for trial in range(30):
        T = 9
        s = r.integers(0, 4, T).astype(float)  # many exact ties
        prot = np.zeros(T, bool)
        prot[0] = True
        prot[r.integers(1, T)] = True
        cand = [t for t in range(T) if not prot[t]]
        k = int(r.integers(0, len(cand) + 1))
        found = []
        for sub in itertools.combinations(cand, k):
            rest = [t for t in cand if t not in sub]
            if all((s[a] > s[b]) or (s[a] == s[b] and a < b) for a in sub for b in rest):
                found.append(sub)
        assert len(found) == 1
        R, _ = O.select_topk(s, k, prot)
        assert R.tolist() == sorted(list(found[0]) + np.nonzero(prot)[0].tolist())


def test_compress_stagewise_brute_force():
    """Each stage of the two-stage prefill recomputed independently: library
    attention for the scores, exhaustive top-k, explicit evicted rows for the
    moments, the finite-difference affine model for the residual."""
    r = rng(18)
    T, d, g, w, B = 40, 6, 2, 4, 14
    K = r.standard_normal((T, d)) * 1.5
    V = r.standard_normal((T, d))
    Q = r.standard_normal((g, w, d)) * 2
    res = O.compress(K, V, Q, B, w, sink=1, keep_window=True, pool=1, mi=True)
    mask = np.zeros((w, T), bool)
    for i in range(w):
        mask[i, :T - w + i + 1] = True
    s = sum(attn_weights(Q[h], K, mask).sum(axis=0) for h in range(g))
    np.testing.assert_allclose(res.scores, s, atol=1e-12)
    prot = np.zeros(T, bool); prot[0] = True; prot[T - w:] = True
    k = B - prot.sum()

    def top(x):
        cand = [t for t in range(T) if not prot[t]]
        order = sorted(cand, key=lambda t: (-x[t], t))
        return np.sort(np.concatenate([np.nonzero(prot)[0], order[:k]]))

    R0 = top(s)
    assert res.idx_stage1.tolist() == R0.tolist()
    E0 = np.setdiff1d(np.arange(T), R0)
    f0 = sdpa(np.zeros(d), K[E0], V[E0])[0]
    J = fd_jacobian_at_zero(K[E0], V[E0])
    rr = V - f0 - K @ J.T
    score2 = s * np.linalg.norm(rr, axis=1)
    np.testing.assert_allclose(res.score2, score2, rtol=1e-6, atol=1e-9)
    R = top(score2)
    assert res.idx.tolist() == R.tolist()
    E = np.setdiff1d(np.arange(T), R)
    sums = (0, np.zeros(d), np.zeros(d), np.zeros((d, d)))
    for t in E:
        sums = O.add_token_sums(sums, K[t], V[t])
    mm = O.from_sums(*sums)
    assert res.moments.n == len(E) == T - B
    np.testing.assert_allclose(res.moments.C, mm.C, atol=1e-12)
    np.testing.assert_allclose(res.moments.mu_k, mm.mu_k, atol=1e-12)
    # mi off = stage 1 only (the SnapKV selection)
    res0 = O.compress(K, V, Q, B, w, mi=False)
    assert res0.idx.tolist() == R0.tolist()
    # nothing evicted when the budget covers the context
    full = O.compress(K, V, Q, T, w)
    assert full.idx.tolist() == list(range(T)) and full.moments.n == 0


def test_select_topk_joint_exhaustive():
    """Joint selection over heads: the unique k-subset of unprotected (head,
    position) pairs whose members all precede every rejected pair in (higher
    score, lower head, lower position) order; one head is select_topk."""
    r = rng(19)
    for trial in range(20):
        H, T = 2, 6
        s = r.integers(0, 3, (H, T)).astype(float)
        prot = np.zeros((H, T), bool)
        prot[:, 0] = True
        cand = [(h, t) for h in range(H) for t in range(T) if not prot[h, t]]
        k = int(r.integers(0, len(cand) + 1))
        found = []
        for sub in itertools.combinations(cand, k):
            rest = [c for c in cand if c not in sub]
            if all((s[a] > s[b]) or (s[a] == s[b] and a < b) for a in sub for b in rest):
                found.append(sub)
        assert len(found) == 1
        R, _ = O.select_topk_joint(s, k, prot)
        for h in range(H):
            want = sorted([t for (hh, t) in found[0] if hh == h] + np.nonzero(prot[h])[0].tolist())
            assert R[h].tolist() == want
    s1 = r.standard_normal((1, 12))
    p1 = np.zeros((1, 12), bool); p1[0, :2] = True
    R, _ = O.select_topk_joint(s1, 5, p1)
    assert R[0].tolist() == O.select_topk(s1[0], 5, p1[0])[0].tolist()


def test_compress_adaptive_reductions_and_stages():
    """Adaptive allocation: one head is `compress`; with several heads the
    stages are recomputed from library attention, explicit evicted rows and
    an independent joint sort; the layer keeps H * budget rows in total."""
    r = rng(20)
    T, d, g, w, B, H = 36, 5, 2, 4, 12, 3
    K = r.standard_normal((H, T, d)) * np.array([0.5, 1.5, 3.0])[:, None, None]
    V = r.standard_normal((H, T, d))
    Q = r.standard_normal((H, g, w, d)) * 2
    one = O.compress_adaptive(K[:1], V[:1], Q[:1], B, w, mi=True)
    ref = O.compress(K[0], V[0], Q[0], B, w, mi=True)
    assert one.idx[0].tolist() == ref.idx.tolist()
    np.testing.assert_allclose(one.moments[0].C, ref.moments.C, atol=1e-12)
    res = O.compress_adaptive(K, V, Q, B, w, mi=True)
    mask = np.zeros((w, T), bool)
    for i in range(w):
        mask[i, :T - w + i + 1] = True
    s = np.stack([sum(attn_weights(Q[h, j], K[h], mask).sum(axis=0) for j in range(g)) for h in range(H)])
    np.testing.assert_allclose(res.scores, s, atol=1e-12)
    prot = np.zeros((H, T), bool); prot[:, 0] = True; prot[:, T - w:] = True
    k = H * B - int(prot.sum())

    def top(x):
        cand = [(h, t) for h in range(H) for t in range(T) if not prot[h, t]]
        order = sorted(cand, key=lambda c: (-x[c], c[0], c[1]))[:k]
        return [sorted([t for (hh, t) in order if hh == h] + np.nonzero(prot[h])[0].tolist()) for h in range(H)]

    R0 = top(s)
    assert [x.tolist() for x in res.idx_stage1] == R0
    score2 = np.zeros((H, T))
    for h in range(H):
        E0 = np.setdiff1d(np.arange(T), R0[h])
        f0 = sdpa(np.zeros(d), K[h][E0], V[h][E0])[0]
        J = fd_jacobian_at_zero(K[h][E0], V[h][E0])
        score2[h] = s[h] * np.linalg.norm(V[h] - f0 - K[h] @ J.T, axis=1)
    np.testing.assert_allclose(res.score2, score2, rtol=1e-6, atol=1e-9)
    R = top(score2)
    assert [x.tolist() for x in res.idx] == R
    assert sum(len(x) for x in R) == H * B
    assert len({len(x) for x in R}) > 1  # the budget moved between heads
    for h in range(H):
        E = np.setdiff1d(np.arange(T), R[h])
        sums = (0, np.zeros(d), np.zeros(d), np.zeros((d, d)))
        for t in E:
            sums = O.add_token_sums(sums, K[h][t], V[h][t])
        mm = O.from_sums(*sums)
        assert res.moments[h].n == len(E)
        np.testing.assert_allclose(res.moments[h].C, mm.C, atol=1e-12)


# --------------------------------------------------------------------------
# Phase 1 (Algorithm 1)
# --------------------------------------------------------------------------

def test_evict_append_brute_force():
    """Every iteration recomputed from explicit rows: alpha from library
    attention summed over the group, residual from the finite-difference
    affine model of the explicit evicted set (empty set: r = v)."""
    r = rng(19)
    d, g, L, budget = 5, 2, 9, 4
    K_R = r.standard_normal((L, d)) * 1.2
    V_R = r.standard_normal((L, d))
    pos = np.arange(100, 100 + L)
    q = r.standard_normal((g, d)) * 2
    kn, vn = r.standard_normal(d), r.standard_normal(d)
    for K_E0, V_E0 in ((np.zeros((0, d)), np.zeros((0, d))),
                       (r.standard_normal((7, d)), r.standard_normal((7, d)))):
        res = O.evict_append(q, K_R, V_R, pos, O.moments_of(K_E0, V_E0), budget,
                             k_new=kn, v_new=vn, pos_new=500)
        Kc, Vc, pc = list(K_R) + [kn], list(V_R) + [vn], list(pos) + [500]
        KE, VE = list(K_E0), list(V_E0)
        expect = []
        while len(Kc) > budget:
            Kr, Vr = np.array(Kc), np.array(Vc)
            alpha = attn_weights(q, Kr).sum(axis=0)
            if KE:
                f0 = sdpa(np.zeros(d), np.array(KE), np.array(VE))[0]
                J = fd_jacobian_at_zero(np.array(KE), np.array(VE))
                rr = Vr - f0 - Kr @ J.T
            else:
                rr = Vr
            sc = alpha * np.linalg.norm(rr, axis=1)
            j = int(np.argmin(sc))
            expect.append(pc[j])
            KE.append(Kc.pop(j)); VE.append(Vc.pop(j)); pc.pop(j)
        assert res.evicted_pos == expect
        assert res.pos.tolist() == pc
        mm = O.moments_of(np.array(KE), np.array(VE))
        assert res.moments.n == len(KE)
        np.testing.assert_allclose(res.moments.C, mm.C, atol=1e-12)
        np.testing.assert_allclose(res.moments.mu_v, mm.mu_v, atol=1e-12)


def test_evict_zero_value_token_goes_first():
    """With no evicted tokens r_j = v_j, so a zero value row has score 0."""
    r = rng(20)
    d = 8
    K, V = r.standard_normal((6, d)), r.standard_normal((6, d))
    V[3] = 0.0
    res = O.evict_append(r.standard_normal((1, d)), K, V, np.arange(6), O.Moments.zeros(d), 5)
    assert res.evicted_pos == [3]
    # exact ties: the lower position is evicted
    V[1] = 0.0
    res = O.evict_append(r.standard_normal((1, d)), K, V, np.arange(6), O.Moments.zeros(d), 5)
    assert res.evicted_pos == [1]


def test_clamp_threshold():
    """App. C.2: S_tilde entries below tau in magnitude are zeroed before use."""
    S = np.array([[1e-7, -2e-6], [5e-7, 3.0]])
    np.testing.assert_array_equal(O.clamp_s_tilde(S, 1e-6), [[0, -2e-6], [0, 3.0]])
    np.testing.assert_array_equal(O.clamp_s_tilde(S, 0.0), S)
    # the threshold applies to S_tilde = n C, not to C: with n = 1000 an entry
    # C_ab = 4e-9 (S_tilde_ab = 4e-6) survives, C_ab = 4e-10 (4e-7) is zeroed
    d, n = 4, 1000
    C = np.zeros((d, d)); C[1, 2] = 4e-9; C[2, 3] = 4e-10
    m = O.Moments(n, np.zeros(d), np.zeros(d), C)
    q = np.array([0.0, 0.0, 1.0, 1.0])
    expect = np.array([0.0, 4e-6 / (n * 2.0), 0.0, 0.0])   # S_tilde q / (n sqrt(d))
    np.testing.assert_allclose(O.fhat_E(q, m, tau=1e-6), expect, rtol=1e-12, atol=0)
    np.testing.assert_allclose(O.fhat_E(q, m, tau=0.0), expect + [0, 0, 4e-7 / (n * 2.0), 0],
                               rtol=1e-12, atol=0)
    K = np.array([[0.0, 0.0, 1.0, 1.0]])
    np.testing.assert_allclose(O.residual(K, np.zeros((1, d)), m, tau=1e-6)[0], -expect,
                               rtol=1e-12, atol=0)


# --------------------------------------------------------------------------
# Table 5
# --------------------------------------------------------------------------

def test_storage_matches_table5():
    path = os.path.join(GOLDEN, "table5_moment_storage.txt")
    rows = [l.split() for l in open(path) if l.strip() and not l.startswith("#")]
    assert len(rows) == 2
    for name, layers, heads, d, mb in rows:
        got = O.storage_bytes(int(layers), int(heads), int(d)) / 1e6
        assert round(got, 1) == float(mb), (name, got)
    # "S occupies 128 x 128 x 2 = 32,768 bytes" per head (App. A.1)
    assert O.storage_bytes(1, 1, 128) - 2 * 2 * 128 == 32768
