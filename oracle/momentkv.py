"""MomentKV oracle: plain, slow, fp64 restatement of the method.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import this
module; only the test suite, the smoke check and the CPU-baseline leg of the
benchmark use it.  It shares no code with the CUDA path: it receives the same
bf16-rounded tensors (widened to float64) and recomputes every quantity from
the paper's definitions, in the paper's order, with numpy.

Notation follows the paper: d head dimension, scale = 1/sqrt(d), logits
s_i = q.k_i / sqrt(d); retained set R, evicted set E with n_e = |E|.

Moment representation.  The paper keeps the raw sums (n_e, s_k, s_v, S)
(Sec. 4.1, Eq. app_sufficient).  The library's state is the equivalent
(n, mu_k, mu_v, C) with mu_k = s_k/n, mu_v = s_v/n and
C = S_tilde / n, S_tilde = sum_E v (k - k_bar)^T = S - s_v s_k^T / n
(Eq. app_S_tilde): C is the population value-key cross-covariance, value
index on rows, key index on columns.  `to_sums` / `from_sums` convert.

Every function cites the passage it follows.  Where the paper is silent the
function states the reading it takes.
"""
from __future__ import annotations

import math
from dataclasses import dataclass

import numpy as np

F64 = np.float64


# ---------------------------------------------------------------------------
# Attention and its decomposition (Sec. 2, Eqs. full-attention, sub-outputs,
# decomposition)
# ---------------------------------------------------------------------------

def logits(q, K):
    """s_i = q^T k_i / sqrt(d)  (Sec. 2, notation paragraph)."""
    K = np.asarray(K, F64)
    q = np.asarray(q, F64)
    return K @ q / math.sqrt(K.shape[1])


def log_partition(s):
    """log sum_i exp(s_i), evaluated with the max shifted out; -inf if empty."""
    s = np.asarray(s, F64)
    if s.size == 0:
        return -math.inf
    m = float(s.max())
    return m + math.log(float(np.exp(s - m).sum()))


def full_attention(q, K, V):
    """f(q) = sum_i exp(s_i) v_i / Z  (Eq. full-attention).  Returns (f, log Z)."""
    s = logits(q, K)
    lz = log_partition(s)
    w = np.exp(s - lz)
    return w @ np.asarray(V, F64), lz


def sub_outputs(q, K, V, retained):
    """f_R, Z_R, f_E, Z_E of Eq. sub-outputs, partition functions in log form.

    `retained` is a boolean mask over the rows of K/V.  An empty subset gets
    output None and log-partition -inf.
    """
    retained = np.asarray(retained, bool)
    out = []
    for mask in (retained, ~retained):
        if mask.any():
            f, lz = full_attention(q, np.asarray(K, F64)[mask], np.asarray(V, F64)[mask])
        else:
            f, lz = None, -math.inf
        out.extend([f, lz])
    return tuple(out)  # f_R, logZ_R, f_E, logZ_E


# ---------------------------------------------------------------------------
# Moment statistics (Sec. 4.1 and Appendix A.1)
# ---------------------------------------------------------------------------

@dataclass
class Moments:
    """(n, mu_k, mu_v, C) of one evicted set; C = S_tilde / n (rows: value dims)."""

    n: int
    mu_k: np.ndarray
    mu_v: np.ndarray
    C: np.ndarray

    @staticmethod
    def zeros(d):
        """Moments with no evicted token (Sec. 5.1: statistics start at zero)."""
        return Moments(0, np.zeros(d), np.zeros(d), np.zeros((d, d)))

    def copy(self):
        return Moments(int(self.n), self.mu_k.copy(), self.mu_v.copy(), self.C.copy())


def moments_of(K_E, V_E):
    """Moments of an explicit evicted set, straight from the definitions.

    k_bar = mean of keys, v_bar = mean of values (Sec. 4.1),
    S_tilde = sum_i v_i (k_i - k_bar)^T  (Eq. fhat's covariance, App. A.1),
    C = S_tilde / n_e.
    """
    K_E = np.asarray(K_E, F64)
    V_E = np.asarray(V_E, F64)
    n, d = K_E.shape[0], K_E.shape[1]
    if n == 0:
        return Moments.zeros(d)
    k_bar = K_E.sum(axis=0) / n
    v_bar = V_E.sum(axis=0) / n
    S_tilde = np.zeros((d, d))
    for i in range(n):
        S_tilde += np.outer(V_E[i], K_E[i] - k_bar)
    return Moments(n, k_bar, v_bar, S_tilde / n)


def to_sums(m: Moments):
    """(n, mu_k, mu_v, C) -> raw sums (n_e, s_k, s_v, S) of Eq. app_sufficient.

    s_k = n mu_k, s_v = n mu_v and, inverting Eq. app_S_tilde,
    S = S_tilde + s_v s_k^T / n with S_tilde = n C.
    """
    n = int(m.n)
    if n == 0:
        d = m.mu_k.shape[0]
        return 0, np.zeros(d), np.zeros(d), np.zeros((d, d))
    s_k = n * np.asarray(m.mu_k, F64)
    s_v = n * np.asarray(m.mu_v, F64)
    S = n * np.asarray(m.C, F64) + np.outer(s_v, s_k) / n
    return n, s_k, s_v, S


def recover(n, s_k, s_v, S):
    """k_bar, v_bar, S_tilde from the running sums (App. A.1, recovery identity)."""
    k_bar = s_k / n
    v_bar = s_v / n
    S_tilde = S - np.outer(s_v, s_k) / n
    return k_bar, v_bar, S_tilde


def from_sums(n, s_k, s_v, S):
    """Raw sums -> (n, mu_k, mu_v, C) via the recovery identity (Eq. app_S_tilde)."""
    d = np.asarray(s_k).shape[0]
    if n == 0:
        return Moments.zeros(d)
    k_bar, v_bar, S_tilde = recover(n, np.asarray(s_k, F64), np.asarray(s_v, F64),
                                    np.asarray(S, F64))
    return Moments(int(n), k_bar, v_bar, S_tilde / n)


def add_token_sums(sums, k, v):
    """Eviction update of Eq. app_update: n+=1, s_k+=k, s_v+=v, S+=v k^T."""
    n, s_k, s_v, S = sums
    k = np.asarray(k, F64)
    v = np.asarray(v, F64)
    return n + 1, s_k + k, s_v + v, S + np.outer(v, k)


def add_token_welford(m: Moments, k, v):
    """The same eviction update written on (n, mu_k, mu_v, C).

    Reading (the paper gives only the raw-sum form, Eq. app_update): the
    one-pass Welford form, identical in exact arithmetic,
      n' = n + 1;  dk = k - mu_k;  mu_k' = mu_k + dk / n'
      mu_v' = mu_v + (v - mu_v) / n'
      C' = ((n' - 1) C + (v - mu_v') dk^T) / n'.
    """
    k = np.asarray(k, F64)
    v = np.asarray(v, F64)
    n1 = m.n + 1
    dk = k - m.mu_k
    mu_k = m.mu_k + dk / n1
    mu_v = m.mu_v + (v - m.mu_v) / n1
    C = ((n1 - 1) * m.C + np.outer(v - mu_v, dk)) / n1
    return Moments(n1, mu_k, mu_v, C)


def merge_chan(a: Moments, b: Moments):
    """Pairwise merge of two disjoint sets' moments (Chan, Golub and LeVeque).

    With delta_k = mu_kb - mu_ka, delta_v = mu_vb - mu_va and co-moments
    M = n C:  M = M_a + M_b + (n_a n_b / n) delta_v delta_k^T.
    Equal in exact arithmetic to summing the raw sums of Eq. app_sufficient.
    """
    if a.n == 0:
        return b.copy()
    if b.n == 0:
        return a.copy()
    n = a.n + b.n
    dk = b.mu_k - a.mu_k
    dv = b.mu_v - a.mu_v
    mu_k = a.mu_k + dk * (b.n / n)
    mu_v = a.mu_v + dv * (b.n / n)
    M = a.n * a.C + b.n * b.C + (a.n * b.n / n) * np.outer(dv, dk)
    return Moments(n, mu_k, mu_v, M / n)


def clamp_s_tilde(S_tilde, tau):
    """Entries of S_tilde with |.| < tau become 0 (App. C.2 safeguard, tau=1e-6)."""
    S_tilde = np.array(S_tilde, F64, copy=True)
    if tau > 0:
        S_tilde[np.abs(S_tilde) < tau] = 0.0
    return S_tilde


# ---------------------------------------------------------------------------
# First-order approximation, Jensen estimate, residual (Sec. 4.1, 4.2)
# ---------------------------------------------------------------------------

def centered_logits(q, K_E):
    """delta_i = q^T (k_i - k_bar) / sqrt(d)  (Sec. 4.1, Eq. centered_softmax)."""
    K_E = np.asarray(K_E, F64)
    return (K_E - K_E.mean(axis=0)) @ np.asarray(q, F64) / math.sqrt(K_E.shape[1])


def fhat_E(q, m: Moments, tau=0.0, order=1):
    """f_hat_E(q) = v_bar + S_tilde q / (n_e sqrt(d))  (Eq. fhat).

    order=0 keeps only v_bar (the zeroth-order variant of Table 4).  The
    clamp of App. C.2 is applied to S_tilde = n C before the product.
    """
    d = m.mu_v.shape[0]
    if order == 0:
        return np.array(m.mu_v, F64)
    S_tilde = clamp_s_tilde(m.n * np.asarray(m.C, F64), tau)
    return np.asarray(m.mu_v, F64) + S_tilde @ np.asarray(q, F64) / (m.n * math.sqrt(d))


def log_zhat_E(q, m: Moments):
    """log Z_hat_E = log n_e + q^T k_bar / sqrt(d)  (Eq. jensen)."""
    d = m.mu_k.shape[0]
    return math.log(m.n) + float(np.asarray(q, F64) @ m.mu_k) / math.sqrt(d)


def residual(K, V, m: Moments, tau=0.0):
    """Moment residual r_j = v_j - v_bar - S_tilde k_j / (n_e sqrt(d))  (Eq. residual).

    With no evicted token Algorithm 1 sets v_bar and S_tilde to zero, so
    r_j = v_j.  Rows of the result correspond to rows of K/V.
    """
    K = np.asarray(K, F64)
    V = np.asarray(V, F64)
    if m.n == 0:
        return V.copy()
    d = K.shape[1]
    S_tilde = clamp_s_tilde(m.n * np.asarray(m.C, F64), tau)
    r = np.empty_like(V)
    for j in range(K.shape[0]):
        r[j] = V[j] - m.mu_v - S_tilde @ K[j] / (m.n * math.sqrt(d))
    return r


# ---------------------------------------------------------------------------
# Phase 2: normalisation-corrected inference (Algorithm 1, Eq. fused, App. C.2)
# ---------------------------------------------------------------------------

def corrected_output(q, K_R, V_R, m: Moments, correction=True, order=1, tau=0.0):
    """One query head: returns (out, lse).

    Algorithm 1 Phase 2: f_R, Z_R from attention over R; if n_e = 0 return
    f_R; otherwise Z_hat_E (Eq. jensen), f_hat_E (Eq. fhat) and the mixing
    weight w_R = Z_R / (Z_R + Z_hat_E) (Eq. fused), evaluated in the log
    domain with logsumexp (App. C.2).  `lse` is the log of the normaliser
    the output was divided by: log Z_R, or log(Z_R + Z_hat_E) when the
    correction is applied.
    Readings: with an empty R and n_e > 0 the output is f_hat_E; an empty R
    with n_e = 0 has no defined output (ValueError).
    """
    K_R = np.asarray(K_R, F64)
    V_R = np.asarray(V_R, F64)
    L = K_R.shape[0]
    use_moments = correction and m.n > 0
    if L == 0 and not use_moments:
        raise ValueError("empty retained set and no evicted moments")
    if L > 0:
        f_R, log_Z_R = full_attention(q, K_R, V_R)
    if not use_moments:
        return f_R, log_Z_R
    f_E_hat = fhat_E(q, m, tau=tau, order=order)
    log_Z_E_hat = log_zhat_E(q, m)
    if L == 0:
        return f_E_hat, log_Z_E_hat
    top = max(log_Z_R, log_Z_E_hat)
    lse = top + math.log(math.exp(log_Z_R - top) + math.exp(log_Z_E_hat - top))
    w_R = math.exp(log_Z_R - lse)
    return w_R * f_R + (1.0 - w_R) * f_E_hat, lse


def decode_step(q, K_R, V_R, m: Moments, k_new=None, v_new=None,
                correction=True, order=1, tau=0.0):
    """Decode for one (batch, KV head) unit and its g query heads.

    q: [g, d].  If k_new/v_new are given they are appended to R first
    (Algorithm 1, the step R <- R u {(k_new, v_new)}), then every query head
    takes `corrected_output` over the same R and moments.
    Returns (out [g, d], lse [g], K_R', V_R').
    """
    K_R = np.asarray(K_R, F64)
    V_R = np.asarray(V_R, F64)
    if k_new is not None:
        K_R = np.vstack([K_R, np.asarray(k_new, F64)[None]])
        V_R = np.vstack([V_R, np.asarray(v_new, F64)[None]])
    q = np.asarray(q, F64)
    outs, lses = [], []
    for h in range(q.shape[0]):
        o, l = corrected_output(q[h], K_R, V_R, m, correction, order, tau)
        outs.append(o)
        lses.append(l)
    return np.stack(outs), np.array(lses), K_R, V_R


# ---------------------------------------------------------------------------
# Phase 1: moment-informed eviction (Algorithm 1)
# ---------------------------------------------------------------------------

def group_attention_weights(q, K_R):
    """alpha_j over the retained rows for a group of query heads.

    Algorithm 1 takes alpha = softmax(q^T K_R / sqrt(d)) for one head.
    Reading for grouped-query attention (the paper is single-head): the
    g query heads that share the KV head each give a softmax over R, and
    alpha_j is their sum.
    """
    q = np.atleast_2d(np.asarray(q, F64))
    alpha = np.zeros(np.asarray(K_R).shape[0])
    for h in range(q.shape[0]):
        s = logits(q[h], K_R)
        alpha += np.exp(s - log_partition(s))
    return alpha


@dataclass
class EvictResult:
    K: np.ndarray
    V: np.ndarray
    pos: np.ndarray
    moments: Moments
    evicted_pos: list
    gaps: list  # relative gap between the smallest and second-smallest score


def evict_append(q, K_R, V_R, pos_R, m: Moments, budget, tau=0.0,
                 k_new=None, v_new=None, pos_new=None):
    """Algorithm 1, the append step and Phase 1, literally.

    Optionally append (k_new, v_new) at position pos_new.  Then, while
    |R| > budget: recover k_bar, v_bar, S_tilde from the running sums (or
    zeros if n_e = 0), alpha over R, r_j (Eq. residual), score = alpha_j
    ||r_j||, evict j* = argmin, add it to the sums (Eq. app_update), remove
    it from R.  Ties in the argmin go to the lower position (rows are kept in
    ascending position order, so to the lower row).  The clamp of App. C.2 is
    applied to S_tilde each time it is recovered.
    Returns an EvictResult with the surviving rows in their original order.
    """
    K = [np.asarray(r, F64) for r in np.asarray(K_R, F64)]
    V = [np.asarray(r, F64) for r in np.asarray(V_R, F64)]
    pos = [int(p) for p in np.asarray(pos_R)]
    if k_new is not None:
        K.append(np.asarray(k_new, F64))
        V.append(np.asarray(v_new, F64))
        pos.append(int(pos_new))
    d = np.asarray(m.mu_k).shape[0]
    sums = to_sums(m)
    evicted, gaps = [], []
    while len(K) > budget:
        n_e, s_k, s_v, S = sums
        Kr = np.array(K).reshape(len(K), d)
        Vr = np.array(V).reshape(len(V), d)
        if n_e > 0:
            _, v_bar, S_tilde = recover(n_e, s_k, s_v, S)
            S_tilde = clamp_s_tilde(S_tilde, tau)
        else:
            v_bar, S_tilde = np.zeros(d), np.zeros((d, d))
        alpha = group_attention_weights(q, Kr)
        scores = np.empty(len(K))
        for j in range(len(K)):
            r_j = Vr[j] - v_bar
            if n_e > 0:
                r_j = r_j - S_tilde @ Kr[j] / (n_e * math.sqrt(d))
            scores[j] = alpha[j] * math.sqrt(float(r_j @ r_j))
        j_star = int(np.argmin(scores))  # first minimum = lowest position
        srt = np.sort(scores)
        gaps.append(float((srt[1] - srt[0]) / abs(srt[1])) if len(srt) > 1 and srt[1] != 0 else math.inf)
        sums = add_token_sums(sums, K[j_star], V[j_star])
        evicted.append(pos[j_star])
        del K[j_star], V[j_star], pos[j_star]
    out_m = from_sums(*sums)
    return EvictResult(np.array(K).reshape(len(K), d), np.array(V).reshape(len(V), d),
                       np.array(pos, np.int64), out_m, evicted, gaps)


# ---------------------------------------------------------------------------
# Prefill compress (Sec. 5.1 SnapKV protocol + the moment-alignment filter)
# ---------------------------------------------------------------------------

def window_scores(Q_obs, K, causal=True):
    """Observation-window scores of the SnapKV prefill protocol (Sec. 5.1).

    Q_obs: [g, w, d], the last w queries of each of the g query heads that
    share this KV head; K: [T, d].  Window query i sits at position T-w+i and,
    when causal, sees keys t <= T-w+i.  Each (head, query) row is a softmax
    over its visible keys; a token's score is the sum of its probabilities
    over all g*w rows.
    """
    Q_obs = np.asarray(Q_obs, F64)
    K = np.asarray(K, F64)
    g, w, _ = Q_obs.shape
    T = K.shape[0]
    s = np.zeros(T)
    for h in range(g):
        for i in range(w):
            visible = T - w + i + 1 if causal else T
            lg = logits(Q_obs[h, i], K[:visible])
            s[:visible] += np.exp(lg - log_partition(lg))
    return s


def pool_scores(s, pool):
    """Merge adjacent tokens into aligned chunks of `pool` (Sec. 5.1, size 4).

    Reading: non-overlapping chunks [c*pool, (c+1)*pool); every token takes
    its chunk's summed score.  pool=1 leaves the scores unchanged.
    """
    s = np.asarray(s, F64)
    if pool <= 1:
        return s.copy()
    out = np.empty_like(s)
    for c0 in range(0, s.shape[0], pool):
        out[c0:c0 + pool] = s[c0:c0 + pool].sum()
    return out


def protected_mask(T, window, sink, keep_window):
    """Sink tokens {0..sink-1} and, if kept, the window {T-w..T-1} (Sec. 5.1)."""
    m = np.zeros(T, bool)
    m[:min(sink, T)] = True
    if keep_window:
        m[max(0, T - window):] = True
    return m


def select_topk(scores, k, protected):
    """R = protected u the k highest-scoring unprotected positions.

    Order: higher score first, equal scores -> lower position first.
    Returns (sorted positions of R, relative gap at the boundary) where the
    gap is (x_k - x_{k+1}) / |x_k| between the last selected and the first
    rejected candidate (inf when nothing is rejected or selected).
    """
    scores = np.asarray(scores, F64)
    cand = np.nonzero(~protected)[0]
    order = sorted(cand.tolist(), key=lambda t: (-scores[t], t))
    chosen = order[:k]
    gap = math.inf
    if 0 < k < len(order):
        a, b = scores[order[k - 1]], scores[order[k]]
        gap = (a - b) / abs(a) if a != 0 else (0.0 if b == a else math.inf)
    R = np.sort(np.concatenate([np.nonzero(protected)[0], np.array(chosen, np.int64)]))
    return R.astype(np.int64), gap


@dataclass
class CompressResult:
    idx: np.ndarray          # retained positions, ascending
    moments: Moments         # of E = all \ R
    scores: np.ndarray       # stage-1 (pooled) window scores s_t
    idx_stage1: np.ndarray   # R0
    score2: np.ndarray | None
    gap1: float
    gap2: float | None


def compress(K, V, Q_obs, budget, window, sink=1, keep_window=True, pool=1,
             mi=True, tau=0.0, causal=True):
    """Prefill compression of one (batch, KV head) unit.

    Reading of how moment-informed eviction enters the prefill (the paper
    runs Algorithm 1 one eviction at a time and only says it adopts the
    SnapKV protocol, Sec. 5.1): two data-parallel stages.
      1. s = window scores (pooled); R0 = protected u top-k(s),
         k = budget - |protected|.
      2. (mi) M0 = moments of E0 = all \\ R0; r_t = Eq. residual under M0;
         score2_t = s_t ||r_t|| (Algorithm 1's score with alpha = s);
         R = protected u top-k(score2).
    The output moments are those of E = all \\ R, taken from the
    definitions.  With T <= budget nothing is evicted.
    """
    K = np.asarray(K, F64)
    V = np.asarray(V, F64)
    T, d = K.shape
    s = pool_scores(window_scores(Q_obs, K, causal), pool)
    if T <= budget:
        return CompressResult(np.arange(T), Moments.zeros(d), s, np.arange(T), None,
                              math.inf, None)
    prot = protected_mask(T, window, sink, keep_window)
    k = budget - int(prot.sum())
    if k < 0:
        raise ValueError("budget smaller than the protected set")
    R0, gap1 = select_topk(s, k, prot)
    R, score2, gap2 = R0, None, None
    if mi:
        keep0 = np.zeros(T, bool)
        keep0[R0] = True
        M0 = moments_of(K[~keep0], V[~keep0])
        r = residual(K, V, M0, tau)
        score2 = s * np.sqrt((r * r).sum(axis=1))
        R, gap2 = select_topk(score2, k, prot)
    keep = np.zeros(T, bool)
    keep[R] = True
    return CompressResult(R, moments_of(K[~keep], V[~keep]), s, R0, score2, gap1, gap2)


def select_topk_joint(scores, k, protected):
    """Adaptive budget across heads (Ada-KV allocation, Sec. 5.1): R_h =
    protected_h u the k highest-scoring unprotected (head, position) pairs of
    all heads together.

    scores, protected: [H, T].  Order: higher score first, equal scores ->
    lower head, then lower position first.  Returns (list of sorted R_h, gap
    at the joint boundary as in select_topk).
    """
    scores = np.asarray(scores, F64)
    H, T = scores.shape
    cand = [(h, t) for h in range(H) for t in range(T) if not protected[h, t]]
    order = sorted(cand, key=lambda ht: (-scores[ht], ht[0], ht[1]))
    chosen = order[:k]
    gap = math.inf
    if 0 < k < len(order):
        a, b = scores[order[k - 1]], scores[order[k]]
        gap = (a - b) / abs(a) if a != 0 else (0.0 if b == a else math.inf)
    keep = np.asarray(protected, bool).copy()
    for h, t in chosen:
        keep[h, t] = True
    return [np.nonzero(keep[h])[0].astype(np.int64) for h in range(H)], gap


@dataclass
class CompressAdaptiveResult:
    idx: list                # per head: retained positions, ascending
    moments: list            # per head: Moments of E_h = all \ R_h
    scores: np.ndarray       # [H, T] stage-1 (pooled) window scores
    idx_stage1: list         # per head: R0_h
    score2: np.ndarray | None
    gap1: float
    gap2: float | None


def compress_adaptive(K, V, Q_obs, budget, window, sink=1, keep_window=True, pool=1,
                      mi=True, tau=0.0, causal=True):
    """Prefill compression of the H KV heads of one layer with the budget
    allocated across heads (the paper's protocol builds on Ada-KV: the layer's
    budget H * budget is shared by the heads according to their attention
    mass, Sec. 5.1).

    K, V: [H, T, d]; Q_obs: [H, g, w, d].  Reading: both selection stages of
    `compress` become joint top-k over the heads' unprotected positions, with
    k = H * budget - sum_h |protected_h| (select_topk_joint); every head keeps
    its own protected set; M0_h and the output moments are per head.  With
    T <= budget every head keeps everything.
    """
    K = np.asarray(K, F64)
    V = np.asarray(V, F64)
    H, T, d = K.shape
    s = np.stack([pool_scores(window_scores(Q_obs[h], K[h], causal), pool) for h in range(H)])
    if T <= budget:
        all_idx = [np.arange(T) for _ in range(H)]
        return CompressAdaptiveResult(all_idx, [Moments.zeros(d) for _ in range(H)], s, all_idx, None,
                                      math.inf, None)
    prot = np.stack([protected_mask(T, window, sink, keep_window) for _ in range(H)])
    k = H * budget - int(prot.sum())
    if k < 0:
        raise ValueError("budget smaller than the protected set")
    R0, gap1 = select_topk_joint(s, k, prot)
    R, score2, gap2 = R0, None, None
    if mi:
        score2 = np.zeros((H, T))
        for h in range(H):
            keep0 = np.zeros(T, bool)
            keep0[R0[h]] = True
            M0 = moments_of(K[h][~keep0], V[h][~keep0])
            r = residual(K[h], V[h], M0, tau)
            score2[h] = s[h] * np.sqrt((r * r).sum(axis=1))
        R, gap2 = select_topk_joint(score2, k, prot)
    moms = []
    for h in range(H):
        keep = np.zeros(T, bool)
        keep[R[h]] = True
        moms.append(moments_of(K[h][~keep], V[h][~keep]))
    return CompressAdaptiveResult(R, moms, s, R0, score2, gap1, gap2)


# ---------------------------------------------------------------------------
# Diagnostics used by the pins (Sec. 3; Appendix A.2, B)
# ---------------------------------------------------------------------------

def error_bound(q, K_E, V_E):
    """Leading term of Eq. app_error_bound: sigma^2 e^sigma / 2 (V_max + ||f_hat_E||)."""
    delta = centered_logits(q, K_E)
    sigma = float(np.abs(delta).max())
    vmax = float(np.sqrt((np.asarray(V_E, F64) ** 2).sum(axis=1)).max())
    fh = fhat_E(q, moments_of(K_E, V_E))
    return 0.5 * sigma * sigma * math.exp(sigma) * (vmax + float(np.linalg.norm(fh))), sigma


def storage_bytes(n_layers, n_kv_heads, d, bytes_per_value=2):
    """Moment storage L_layers * H * (d^2 + 2d) * bytes (App. A.1, Table 5)."""
    return n_layers * n_kv_heads * (d * d + 2 * d) * bytes_per_value
