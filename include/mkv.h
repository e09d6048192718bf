/*
 * mkv.h -- C ABI of the MomentKV hot path on one GB300 (sm_103a).
 *
 * MomentKV (arXiv 2606.01563) keeps, for every attention head, a summary of
 * the KV pairs evicted from the cache -- the count n, key mean mu_k, value
 * mean mu_v and value-key cross-covariance C -- and uses it twice: to choose
 * which tokens to evict (moment residual, Eq. residual) and to add back a
 * closed-form first-order estimate of the evicted tokens' attention output
 * (Eqs. fhat, jensen, fused).  Four calls cover the data-parallel path:
 *
 *   mkv_compress      prefill: window scores, budget top-k, moment filter,
 *                     evicted-set moments                    (Sec. 5.1, 4.2)
 *   mkv_decode_step   attention over the retained cache merged with the
 *                     moment term in one normaliser     (Algorithm 1 Phase 2)
 *   mkv_evict_append  append a token and evict one at a time down to the
 *                     budget by the moment-informed score (Algorithm 1 Phase 1)
 *   mkv_decode_evict_step  the whole of Algorithm 1 for one generated token:
 *                     append, Phase 1 down to the budget, Phase 2 (continuous
 *                     per-token eviction)
 *
 * Conventions shared by every call
 *  - Pointers are DEVICE pointers unless a comment says otherwise; the
 *    caller allocates and owns every buffer.  The library never allocates or
 *    frees device memory.
 *  - bf16 tensors are IEEE bfloat16 stored as 16-bit words; fp32 is IEEE
 *    binary32.  All tensors are dense, row-major, with the shapes given.
 *  - Index conventions: b batch, h_kv KV head, g = group (query heads per KV
 *    head), query head j uses KV head j / g, d = head_dim in {64, 128},
 *    scale = 1/sqrt(d).  A "unit" is one (batch, KV head) pair.
 *  - Calls are asynchronous and ordered on `stream` (a cudaStream_t; NULL is
 *    the legacy default stream).  Host-side validation failures return an
 *    error and launch nothing.  Errors the kernels detect (capacity overflow
 *    on append, empty attention, a bounded wait that ran out) are written to
 *    an error word inside the workspace and read by mkv_get_device_error.
 *  - A workspace serves one stream at a time; two calls that overlap on the
 *    GPU must not share one.
 */
#ifndef MKV_H
#define MKV_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define MKV_API __attribute__((visibility("default")))
#else
#define MKV_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  MKV_OK = 0,
  MKV_ERR_INVALID_ARG = 1, /* null pointer, bad parameter, empty attention  */
  MKV_ERR_SHAPE = 2,       /* unsupported or inconsistent sizes             */
  MKV_ERR_CAPACITY = 3,    /* cache capacity too small                      */
  MKV_ERR_CUDA = 4,        /* a CUDA runtime call failed                    */
  MKV_ERR_TIMEOUT = 5,     /* a bounded device-side wait ran out            */
  MKV_ERR_UNSUPPORTED = 6, /* head_dim or group outside the built kernels   */
  MKV_ERR_WORKSPACE = 7    /* workspace missing, too small or misaligned    */
} mkv_status;

/* Attention geometry of one layer.  head_dim in {64, 128}; group in {1,2,4,8};
 * 1 <= batch <= 65535 and 1 <= n_kv_heads <= 65535 (grid dimensions of the
 * kernels), batch * n_kv_heads <= 65535 * 64, and for mkv_compress
 * batch * n_kv_heads <= 65535.  Others return MKV_ERR_SHAPE. */
typedef struct {
  int32_t batch;
  int32_t n_kv_heads;
  int32_t group;
  int32_t head_dim;
} mkv_geom;

/*
 * Evicted-set moments, one set per unit (Sec. 4.1, App. A.1).
 *   n    int32 [b, h_kv]          number of evicted tokens n_e
 *   mu_k fp32  [b, h_kv, d]       key mean    k_bar = s_k / n_e
 *   mu_v fp32  [b, h_kv, d]       value mean  v_bar = s_v / n_e
 *   C    fp32  [b, h_kv, d, d]    C[a][c] = S_tilde[a][c] / n_e with
 *                                 S_tilde = sum_E v (k - k_bar)^T (Eq. app_S_tilde):
 *                                 row a indexes value dims, column c key dims.
 * n = 0 means "no evicted token" (the other fields are then ignored); a
 * zero-filled struct is the state at the start of a generation (Sec. 5.1).
 * Alignment: mu_k 8 bytes, mu_v and C 16 bytes (the kernels read them with
 * vector loads); a misaligned pointer is rejected with MKV_ERR_INVALID_ARG
 * before anything is launched.
 */
typedef struct {
  int32_t* n;
  float* mu_k;
  float* mu_v;
  float* C;
} mkv_moments;

/*
 * Retained KV cache, one slab per unit.
 *   K, V  bf16  [b, h_kv, capacity, d]   rows 0..len-1 are in use
 *   pos   int32 [b, h_kv, capacity]      absolute position of each row; rows
 *                                        are kept in ascending position order
 *   len   int32 [b, h_kv]                rows in use
 *   seen  int32 [b, h_kv]                tokens seen so far; an appended token
 *                                        takes position `seen`, then seen += 1
 * Optional eviction state (both NULL, or both set):
 *   y     fp32  [b, h_kv, capacity, d]   y_j = S_tilde k_j of each row under
 *                                        the current moments (the products
 *                                        Algorithm 1's residual needs), 16-byte
 *                                        aligned
 *   y_len int32 [b, h_kv]                rows 0..y_len-1 of y are current
 * With them, mkv_evict_append and mkv_decode_evict_step compute S_tilde k_j
 * only for rows at or above y_len (the rows appended since the last
 * eviction), O(d^2) each, instead of for every row, and leave y current for
 * the surviving rows; mkv_compress sets y_len to 0.  Appends by
 * mkv_decode_step need no update (they add rows above y_len).  A caller that
 * changes the cache or the moments in any other way sets y_len to 0.
 * Capacities above 1152 rows run an eviction kernel that does not keep y: it
 * sets y_len to 0.
 */
typedef struct {
  void* K;
  void* V;
  int32_t* pos;
  int32_t* len;
  int32_t* seen;
  int32_t capacity;
  float* y;
  int32_t* y_len;
} mkv_cache;

/* Prefill compression parameters (SnapKV protocol of Sec. 5.1 plus the
 * moment filter of Sec. 4.2). */
typedef struct {
  int32_t budget;      /* L: rows kept per unit (includes sink and window)   */
  int32_t window;      /* w: observation window = the last w positions        */
  int32_t sink;        /* leading positions always kept (the paper keeps 1)   */
  int32_t keep_window; /* 1: the w window positions are always kept           */
  int32_t pool;        /* adjacent-token chunk size for scores: 1 (off), 2, 4, 8, 16 or 32 (Sec. 5.1 uses 4) */
  int32_t mi;          /* 1: moment-informed second stage; 0: window scores only */
  int32_t causal;      /* 1: window query i (position T-w+i) sees keys t <= T-w+i */
  float tau;           /* clamp |S_tilde_ab| < tau to 0 in the residual (App. C.2) */
  int32_t adaptive;    /* 1: the layer's budget h_kv * budget is shared by the KV */
                       /* heads of each batch item (Ada-KV allocation, Sec. 5.1): */
                       /* both selections take the top of all heads' unprotected  */
                       /* (head, position) pairs together; 0: budget per unit    */
} mkv_compress_params;

/* Optional outputs of mkv_compress for inspection; any field may be NULL. */
typedef struct {
  float* scores;       /* fp32 [b, h_kv, T] pooled window scores s_t               */
  float* score2;       /* fp32 [b, h_kv, T] s_t * ||r_t|| (mi=1); protected rows 0 */
  int32_t* idx_stage1; /* int32 [b, h_kv, budget] first-stage retained positions;   */
                       /* with adaptive, [b, h_kv * budget] of h * T + t, ascending */
} mkv_compress_diag;

/* Decode parameters (Algorithm 1 Phase 2, Table 4, App. C.2). */
typedef struct {
  int32_t correction; /* 1: merge the moment term; 0: plain attention over R   */
  int32_t order;      /* 1: f_hat_E = v_bar + S_tilde q/(n sqrt d); 0: v_bar only */
  float tau;          /* clamp |S_tilde_ab| < tau to 0 before S_tilde q         */
  const void* C16;    /* optional bf16 [b, h_kv, d, d] copy of the moments' C   */
                      /* (16-bit moment storage, Sec. C.2; mkv_moments_pack_bf16): */
                      /* when set, the order-1 term reads C from it (half the  */
                      /* bytes) instead of mkv_moments.C; 16-byte aligned.     */
  int32_t early_load; /* 1: the caller guarantees that no kernel which may still */
                      /* run when this call's kernel starts writes this cache   */
                      /* or these moments: in a model's layer chain, the        */
                      /* previous layer's kernels (and, if the preceding kernel */
                      /* releases its dependents before waiting on its own      */
                      /* predecessor, that predecessor too).  The kernel then   */
                      /* reads the cache length and moment rows and starts the  */
                      /* first tile copies before its programmatic dependency   */
                      /* wait, overlapping the preceding kernel; only q, k_new  */
                      /* and v_new are read after it.  A length that changed in */
                      /* between is recorded as MKV_ERR_INVALID_ARG (outputs    */
                      /* undefined); other violations go undetected.  0: every */
                      /* read waits (always safe).  mkv_decode_evict_step        */
                      /* ignores it (its own eviction kernel writes the cache). */
  const void* C_split; /* optional [b, h_kv, d, d/2] pairs of 32-bit words from  */
                       /* mkv_moments_pack_split: C' of Eq. fused (C with the     */
                       /* App. C.2 clamp applied) split into bf16 hi and lo      */
                       /* parts.  When set, the order-1 term reads it instead of */
                       /* mkv_moments.C: the same bytes, and the same products,  */
                       /* without the clamp and split at every step.  Valid     */
                       /* while the moments and tau are those of the pack (the  */
                       /* output is then bit-identical to the fp32-C path); not  */
                       /* with C16; 16-byte aligned.                             */
} mkv_decode_params;

/*
 * 16-bit moment storage (Sec. C.2 keeps the moments in 16 bits): writes
 * C16[u] = bf16(mom->C[u]) (round to nearest even) for every unit, one launch
 * on `stream`.  C16 is caller-owned device memory of b * h_kv * d * d bf16,
 * 16-byte aligned; pass it as mkv_decode_params.C16.  Returns
 * MKV_ERR_INVALID_ARG on null or misaligned pointers.
 */
MKV_API mkv_status mkv_moments_pack_bf16(mkv_geom geom, const mkv_moments* mom, void* C16, void* stream);

/*
 * The decode's operand form of C' (Eq. fused, App. C.2), written once when the
 * moments change instead of at every decode step: for every unit u, row a
 * and column pair (c, c + 1), with x = C[u][a][c] and y = C[u][a][c + 1]
 * each set to 0 where |n_u x| < tau (the clamp of S_tilde = n C), word 0 is
 * bf16x2(x, y) and word 1 is bf16x2(x - bf16(x), y - bf16(y)) (round to nearest
 * even; the first value in the low half).  One launch on `stream`.  C_split
 * is caller-owned device memory of b * h_kv * d * d 32-bit words (as many bytes
 * as C), 16-byte aligned; pass it as mkv_decode_params.C_split with the same
 * tau, and pack again after every call that changes the moments
 * (mkv_compress, mkv_evict_append).  Returns MKV_ERR_INVALID_ARG on null or
 * misaligned pointers or a negative or NaN tau.
 */
MKV_API mkv_status mkv_moments_pack_split(mkv_geom geom, const mkv_moments* mom, float tau, void* C_split,
                                          void* stream);

/* Human-readable name of a status code (static string). */
MKV_API const char* mkv_status_str(mkv_status s);

/* Library ABI version (major * 10000 + minor * 100 + patch). */
MKV_API int32_t mkv_version(void);

/*
 * Bytes of device workspace mkv_compress needs for this geometry and T.
 * Returns 0 if the arguments are invalid.  The workspace needs no
 * initialisation.
 */
MKV_API size_t mkv_compress_workspace_size(mkv_geom geom, int32_t T, const mkv_compress_params* p);

/*
 * Prefill compression of one layer (Sec. 5.1 protocol, Sec. 4.2 moments).
 *   K, V   bf16 [b, h_kv, T, d]       keys and values of the whole prompt
 *   Q_obs  bf16 [b, h_kv, g, w, d]    the last w queries of each query head
 * Per unit:
 *   1. logits l_{h,i,t} = scale q_{h,i} . k_t over the g*w window rows
 *      (causal: row i sees t <= T-w+i); s_t = sum over rows of softmax; pooled
 *      into aligned chunks of `pool` tokens.
 *   2. R0 = protected (sink, and the window if keep_window) plus the
 *      budget-|protected| highest s_t; ties keep the lower position.
 *   3. if mi: moments M0 of E0 = all \ R0; r_t = v_t - mu_v0 - scale C0' k_t
 *      with C0' = C0 clamped where |n0 C0| < tau (Eq. residual); score2 =
 *      s_t ||r_t||; R = protected plus the top of score2, same tie rule.
 *      if !mi: R = R0.
 *   4. writes the retained rows of R to out_cache in ascending position
 *      (K, V, pos), len = |R|, seen = T, and the moments of E = all \ R to
 *      out_mom (overwritten).  If T <= budget every token is kept and n = 0.
 * With adaptive = 1 (T > budget), steps 2 and 3 select jointly over the h_kv
 * heads of a batch item: R_h = protected_h plus head h's share of the top
 * h_kv * (budget - |protected|) unprotected (head, position) pairs; ties keep
 * the lower head, then the lower position.  len then differs per head and
 * sums to h_kv * budget over a batch item; rows of out_cache from len up to
 * the next multiple of 128 (below capacity) are overwritten with zeros.
 * Requirements: budget >= sink + (keep_window ? w : 0), 1 <= w <= T,
 * g * w <= 256 window rows (else MKV_ERR_SHAPE),
 * out_cache->capacity >= min(T, budget) (adaptive: >= min(T, h_kv * budget -
 * (h_kv - 1) * |protected|), h_kv <= 64, h_kv * T <= 2^28), T <= 1,048,576.
 */
MKV_API mkv_status mkv_compress(mkv_geom geom, int32_t T, const void* K, const void* V, const void* Q_obs,
                        const mkv_compress_params* p, const mkv_cache* out_cache,
                        const mkv_moments* out_mom, const mkv_compress_diag* diag,
                        void* workspace, size_t workspace_bytes, void* stream);

/*
 * Bytes of device workspace mkv_decode_step needs for this geometry and cache
 * capacity on the current device.  Returns 0 if the arguments are invalid.
 * The workspace must be zero-filled before its first use; every call leaves
 * it ready for the next one.
 */
MKV_API size_t mkv_decode_workspace_size(mkv_geom geom, int32_t capacity);

/*
 * One decode step for every unit (Algorithm 1: append, then Phase 2).
 *   q             bf16 [b, g*h_kv, d]   this step's queries
 *   k_new, v_new  bf16 [b, h_kv, d]     optional (both NULL or both set): the
 *                                       new token is appended at row len with
 *                                       position seen before attending.
 *   out           fp32 [b, g*h_kv, d]   corrected output f_hat(q) (Eq. fused)
 *   lse           fp32 [b, g*h_kv]      optional: natural log of the merged
 *                                       normaliser, log(Z_R + Z_hat_E), or log
 *                                       Z_R when no correction applies.
 * For each query head: (m_R, l_R, o_R) over the retained rows; if
 * correction && n > 0: log Z_hat_E = log n + scale q.mu_k (Eq. jensen),
 * f_hat_E = mu_v + scale C' q (order 1, C' clamped as in mkv_compress) or
 * mu_v (order 0), w_R from a log-sum-exp of log Z_R and log Z_hat_E
 * (App. C.2), out = w_R o_R + (1 - w_R) f_hat_E.  With no retained row the
 * output is f_hat_E; with neither rows nor moments the kernel records
 * MKV_ERR_INVALID_ARG and writes zeros.  An append past capacity records
 * MKV_ERR_CAPACITY, still attends over the new token, and leaves the cache
 * unchanged.  q, out, k_new and v_new must be 16-byte aligned.
 */
MKV_API mkv_status mkv_decode_step(mkv_geom geom, const void* q, const void* k_new, const void* v_new,
                           const mkv_cache* cache, const mkv_moments* mom,
                           const mkv_decode_params* p, float* out, float* lse,
                           void* workspace, size_t workspace_bytes, void* stream);

/*
 * mkv_decode_step without a workspace argument.  The paper has no
 * counterpart: this is a deployment variant for callers that cannot
 * allocate device memory when they decode -- a plugin that its host engine
 * gives only input and output buffers, a server whose device memory another
 * allocator reserved at start-up, or a latency-critical path that cannot
 * accept cudaMalloc's implicit device synchronisation.
 * Arguments, computation and outputs are those of mkv_decode_step.  The
 * split-K scratch (error word, ticket counters, partial states, moment rows)
 * is a fixed 4 MiB device array inside the library, held by every GPU that
 * loads it until the process exits; this call allocates nothing and frees
 * nothing.
 *  - The first call on a device sets up that device (looks up the array's
 *    address, zeroes it, synchronises the device); make that first call before
 *    any stream capture.
 *  - Geometries whose scratch would exceed 4 MiB even with one split per unit
 *    (b * h_kv * g * (d + 4) * 4 bytes plus the moment rows) are rejected with
 *    MKV_ERR_WORKSPACE before anything runs; smaller ones use as many splits
 *    as fit.
 *  - Every call shares the array: calls that overlap on the GPU (e.g. on two
 *    streams) race and give wrong results.  Serialise them.
 *  - Errors the kernel detects are recorded in the array's error word, which
 *    this call does not expose and never clears: the first recorded error
 *    stays set until the process exits.  The outputs in those cases are as
 *    described for mkv_decode_step.
 *  - The array's address is looked up on every call; if it changed (the
 *    library's device code was loaded again, e.g. after cudaDeviceReset) the
 *    set-up above runs again.
 */
MKV_API mkv_status mkv_decode_step_noalloc(mkv_geom geom, const void* q, const void* k_new, const void* v_new,
                                           const mkv_cache* cache, const mkv_moments* mom,
                                           const mkv_decode_params* p, float* out, float* lse, void* stream);

/*
 * Bytes of device workspace mkv_evict_append needs.  Returns 0 if invalid.
 * The workspace needs no initialisation.
 */
MKV_API size_t mkv_evict_workspace_size(mkv_geom geom, int32_t capacity);

/*
 * Algorithm 1's append step and Phase 1 for every unit.
 *   q             bf16 [b, g*h_kv, d]   queries whose attention weights score
 *                                       the rows (alpha_j summed over the g
 *                                       query heads of the unit)
 *   k_new, v_new  bf16 [b, h_kv, d]     optional token appended first
 * Then, while len > budget: recover v_bar and S_tilde = n C from the moments
 * (zero if n = 0), clamp |S_tilde_ab| < tau to 0, alpha = sum over the group
 * of softmax(scale q . k_j) over the current rows, r_j = v_j - v_bar -
 * S_tilde k_j / (n sqrt d), score_j = alpha_j ||r_j||, evict the row with
 * the smallest score (ties: the lower position), fold it into the moments
 * (n+1; the equivalent of Eq. app_update on (n, mu_k, mu_v, C)) and remove
 * it.  Surviving rows keep their ascending position order.
 * Requirements: 0 <= budget, capacity <= 65536 (else MKV_ERR_SHAPE),
 * len + (k_new ? 1 : 0) <= capacity (else the kernel records
 * MKV_ERR_CAPACITY and leaves the unit unchanged).
 */
MKV_API mkv_status mkv_evict_append(mkv_geom geom, const void* q, const void* k_new, const void* v_new,
                            int32_t budget, const mkv_cache* cache, const mkv_moments* mom,
                            float tau, void* workspace, size_t workspace_bytes, void* stream);

/*
 * Bytes of device workspace mkv_decode_evict_step needs for this geometry and
 * cache capacity on the current device.  Returns 0 if the arguments are
 * invalid.  The workspace must be zero-filled before its first use; every
 * call leaves it ready for the next one.
 */
MKV_API size_t mkv_decode_evict_workspace_size(mkv_geom geom, int32_t capacity);

/*
 * One decoding step of Algorithm 1 for every unit: append (k_new, v_new) at
 * row len with position seen, run Phase 1 while len > budget (exactly as
 * mkv_evict_append with tau = p->tau), then Phase 2 over the surviving rows
 * and the updated moments (exactly as mkv_decode_step without a new token:
 * out, lse and p->correction, p->order, p->tau as documented there).  With a
 * budget at or above the new length nothing is evicted, so one call per
 * generated token keeps the cache at the budget once it is reached: the
 * paper's continuous eviction mode.  The eviction and the decode kernels
 * run back to back on `stream` (two launches, one workspace).
 *   q             bf16 [b, g*h_kv, d]   this step's queries (score the rows
 *                                       in Phase 1 and attend in Phase 2)
 *   k_new, v_new  bf16 [b, h_kv, d]     the token appended (both required)
 *   out           fp32 [b, g*h_kv, d]   corrected output
 *   lse           fp32 [b, g*h_kv]      optional, as in mkv_decode_step
 * Requirements: as mkv_evict_append and mkv_decode_step; p->C16 and
 * p->C_split must be NULL (the moments change inside the call).  q, out, k_new and v_new must be
 * 16-byte aligned.
 */
MKV_API mkv_status mkv_decode_evict_step(mkv_geom geom, const void* q, const void* k_new, const void* v_new,
                                 int32_t budget, const mkv_cache* cache, const mkv_moments* mom,
                                 const mkv_decode_params* p, float* out, float* lse,
                                 void* workspace, size_t workspace_bytes, void* stream);

/*
 * Synchronises `stream`, returns the first error a kernel recorded in this
 * workspace since the last call (MKV_OK if none) and clears it.  `info`
 * (host pointer, may be NULL) receives a detail word (e.g. the unit index).
 *
 * MKV_ERR_TIMEOUT: a wait on a tile copy or a tensor-core commit ran out
 * (the poll limit is over a second).  The CTA then stops its pipeline,
 * contributes an empty state, and before it exits waits again, with the full
 * limit, for the copies it issued into its shared memory and for its last
 * commit.  If that wait runs out too, the CTA exits with those copies
 * possibly still in flight; the status stays MKV_ERR_TIMEOUT.  Outputs of the
 * call are undefined after any timeout, and after one whose drain also ran
 * out the CUDA context should not be trusted any more.
 */
MKV_API mkv_status mkv_get_device_error(void* workspace, void* stream, int32_t* info);

#ifdef __cplusplus
}
#endif

#endif /* MKV_H */
