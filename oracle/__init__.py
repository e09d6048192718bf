"""fp64 CPU oracle for MomentKV (TEST INFRASTRUCTURE ONLY).

Imported by the test suite, the smoke check and the CPU-baseline leg of the
benchmark; never by the library.  See `momentkv` for the definitions.

Parity status of each function (what pins it, in tests/test_oracle_pins.py):
  full_attention, sub_outputs, log_partition -- torch scaled_dot_product_attention
  moments_of, to_sums/from_sums, add_token_*, merge_chan -- identity
      S_tilde = S - s_v s_k^T / n (Eq. app_S_tilde), incremental = batch,
      exact-rational brute force
  fhat_E, residual -- first-order Taylor expansion of f_E measured by finite
      differences (Eq. fhat is that expansion about q = 0)
  log_zhat_E -- Jensen bound and its tightness (Eqs. jensen, app_ratio,
      app_logit_var), weight-bias identity (Eq. app_weight_bias)
  corrected_output / decode_step -- n_e = 0 and n_e = 1 special cases against
      library attention, error bound (Eq. app_error_bound), limits of App. B.2
  window_scores, pool_scores -- library softmax attention with one-hot values
  select_topk -- exhaustive check over all subsets on tiny inputs
  evict_append -- brute-force recomputation of every candidate score from the
      definitions, constructed cases with a known answer
  compress -- stage-by-stage brute force on tiny inputs; the two-stage
      reading itself is the library's definition (parity unpinned by the paper
      beyond its parts: the paper does not say how the moment filter enters
      the prefill)
  select_topk_joint -- exhaustive check over all subsets of (head, position)
      pairs on tiny inputs; one head reduces to select_topk
  compress_adaptive -- one head equals `compress`; stage-by-stage brute force
      on tiny inputs; the joint allocation across heads is the library's
      reading of the paper's Ada-KV protocol (Sec. 5.1), pinned only by its
      definition beyond those reductions
  storage_bytes -- Table 5 figures
"""
from .momentkv import *  # noqa: F401,F403
from .momentkv import Moments, CompressResult, CompressAdaptiveResult, EvictResult  # noqa: F401
