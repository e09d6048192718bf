"""The oracle's pins must catch plausible mistakes.

Each case copies the oracle and the pin tests into a temporary directory,
plants one mistake in the copied oracle (a transposed operand, a flipped
sign, a dropped term, a wrong index or tie-break), and checks that the pin
suite then fails.  Runs on the CPU only.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

MUTATIONS = {
    "S_tilde transposed in f_hat_E": (
        "return np.asarray(m.mu_v, F64) + S_tilde @ np.asarray(q, F64)",
        "return np.asarray(m.mu_v, F64) + S_tilde.T @ np.asarray(q, F64)"),
    "residual sign": ("r[j] = V[j] - m.mu_v - S_tilde @ K[j]", "r[j] = V[j] - m.mu_v + S_tilde @ K[j]"),
    "log n_e dropped from Z_hat_E": ("return math.log(m.n) + float", "return 0.0 + float"),
    "Welford uses the old value mean": (
        "C = ((n1 - 1) * m.C + np.outer(v - mu_v, dk)) / n1",
        "C = ((n1 - 1) * m.C + np.outer(v - m.mu_v, dk)) / n1"),
    "causal window off by one": ("visible = T - w + i + 1 if causal else T",
                                 "visible = T - w + i if causal else T"),
    "evict argmax": ("j_star = int(np.argmin(scores))", "j_star = int(np.argmax(scores))"),
    "alpha dropped from the eviction score": ("scores[j] = alpha[j] * math.sqrt",
                                              "scores[j] = 1.0 * math.sqrt"),
    "Chan merge without the cross term": (
        "M = a.n * a.C + b.n * b.C + (a.n * b.n / n) * np.outer(dv, dk)",
        "M = a.n * a.C + b.n * b.C"),
    "top-k ties to the higher position": ("key=lambda t: (-scores[t], t)",
                                          "key=lambda t: (-scores[t], -t)"),
    "mixing weights swapped": ("return w_R * f_R + (1.0 - w_R) * f_E_hat, lse",
                               "return (1.0 - w_R) * f_R + w_R * f_E_hat, lse"),
    "1/sqrt(d) missing from logits": ("return K @ q / math.sqrt(K.shape[1])", "return K @ q"),
    "stage-2 score without s": ("score2 = s * np.sqrt((r * r).sum(axis=1))",
                                "score2 = np.sqrt((r * r).sum(axis=1))"),
    "pooling takes the max": ("out[c0:c0 + pool] = s[c0:c0 + pool].sum()",
                              "out[c0:c0 + pool] = s[c0:c0 + pool].max()"),
    "raw-sum conversion sign": ("S = n * np.asarray(m.C, F64) + np.outer(s_v, s_k) / n",
                                "S = n * np.asarray(m.C, F64) - np.outer(s_v, s_k) / n"),
    "joint top-k ties to the higher head": ("key=lambda ht: (-scores[ht], ht[0], ht[1])",
                                           "key=lambda ht: (-scores[ht], -ht[0], ht[1])"),
    "adaptive budget without the protected rows": ("k = H * budget - int(prot.sum())",
                                                   "k = H * budget"),
    "clamp applied to C instead of S_tilde": (
        "S_tilde = clamp_s_tilde(m.n * np.asarray(m.C, F64), tau)\n    return",
        "S_tilde = m.n * clamp_s_tilde(np.asarray(m.C, F64), tau)\n    return"),
    "co-moment without the key mean": ("S_tilde += np.outer(V_E[i], K_E[i] - k_bar)",
                                       "S_tilde += np.outer(V_E[i], K_E[i])"),
    "window scores not normalised per row": ("s[:visible] += np.exp(lg - log_partition(lg))",
                                             "s[:visible] += np.exp(lg)"),
    "causal mask dropped": ("visible = T - w + i + 1 if causal else T", "visible = T"),
    "protected window one short": ("m[max(0, T - window):] = True", "m[max(0, T - window + 1):] = True"),
    "one sink too many": ("m[:min(sink, T)] = True", "m[:min(sink + 1, T)] = True"),
    "residual without the value mean": ("r[j] = V[j] - m.mu_v - S_tilde @ K[j]", "r[j] = V[j] - S_tilde @ K[j]"),
    "residual with a centred key": ("r[j] = V[j] - m.mu_v - S_tilde @ K[j]",
                                    "r[j] = V[j] - m.mu_v - S_tilde @ (K[j] - m.mu_k)"),
    "Jensen logit sign": ("return math.log(m.n) + float(np.asarray(q, F64) @ m.mu_k)",
                          "return math.log(m.n) - float(np.asarray(q, F64) @ m.mu_k)"),
    "f_hat_E without 1/sqrt(d)": ("S_tilde @ np.asarray(q, F64) / (m.n * math.sqrt(d))",
                                  "S_tilde @ np.asarray(q, F64) / m.n"),
    "order 0 keeps the covariance term": ("if order == 0:\n        return np.array(m.mu_v, F64)",
                                          "if order == -1:\n        return np.array(m.mu_v, F64)"),
    "log-sum-exp without its shift": ("lse = top + math.log(", "lse = math.log("),
    "decode does not append": (
        "        K_R = np.vstack([K_R, np.asarray(k_new, F64)[None]])\n"
        "        V_R = np.vstack([V_R, np.asarray(v_new, F64)[None]])",
        "        pass"),
    "recovery identity sign": ("S_tilde = S - np.outer(s_v, s_k) / n\n    return k_bar",
                               "S_tilde = S + np.outer(s_v, s_k) / n\n    return k_bar"),
    "Welford key-mean step": ("mu_k = m.mu_k + dk / n1", "mu_k = m.mu_k + dk / (n1 + 1)"),
    "Chan mean weighted by the wrong count": ("mu_k = a.mu_k + dk * (b.n / n)", "mu_k = a.mu_k + dk * (a.n / n)"),
    "alpha from the first query head only": (
        "    for h in range(q.shape[0]):\n        s = logits(q[h], K_R)",
        "    for h in range(1):\n        s = logits(q[h], K_R)"),
    "eviction ties to the higher position": ("j_star = int(np.argmin(scores))",
                                             "j_star = len(scores) - 1 - int(np.argmin(scores[::-1]))"),
    "evicted token not added to the sums": ("sums = add_token_sums(sums, K[j_star], V[j_star])", "sums = sums"),
    "M0 from the retained set": ("M0 = moments_of(K[~keep0], V[~keep0])", "M0 = moments_of(K[keep0], V[keep0])"),
    "output moments from the retained set": ("return CompressResult(R, moments_of(K[~keep], V[~keep])",
                                             "return CompressResult(R, moments_of(K[keep], V[keep])"),
    "adaptive M0 from the retained set": ("M0 = moments_of(K[h][~keep0], V[h][~keep0])",
                                          "M0 = moments_of(K[h][keep0], V[h][keep0])"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_mutation(name, tmp_path):
    src = open(os.path.join(ROOT, "oracle", "momentkv.py")).read()
    before, after = MUTATIONS[name]
    assert src.count(before) == 1, "mutation site not found"
    shutil.copytree(os.path.join(ROOT, "oracle"), tmp_path / "oracle")
    os.makedirs(tmp_path / "tests")
    for f in ("conftest.py", "test_oracle_pins.py"):
        shutil.copy(os.path.join(ROOT, "tests", f), tmp_path / "tests" / f)
    shutil.copytree(os.path.join(ROOT, "tests", "golden"), tmp_path / "tests" / "golden")
    (tmp_path / "oracle" / "momentkv.py").write_text(src.replace(before, after))
    r = subprocess.run([sys.executable, "-m", "pytest", "tests/test_oracle_pins.py", "-x", "-q",
                        "-p", "no:cacheprovider"], cwd=tmp_path, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 1, f"pins did not catch: {name}\n{r.stdout[-2000:]}"
