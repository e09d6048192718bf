// C-ABI entry points declared in include/mkv.h: argument validation,
// workspace sizing and kernel dispatch.  No allocation, no global state
// beyond a per-device cache of the SM count.
#include <cuda_runtime.h>

#include "common.cuh"
#include "kernels.h"
#include "validate.h"
#include "../../include/mkv_debug.h"

using namespace mkv;

namespace {

int num_sms_current() {
  static int cache[64] = {0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (dev >= 0 && dev < 64 && cache[dev] > 0) return cache[dev];
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
  if (dev >= 0 && dev < 64) cache[dev] = n;
  return n;
}

int protected_count_host(int T, int W, int sink, int keep_window) {
  const int s = sink < T ? sink : T;
  const int w = keep_window ? (W < T ? W : T) : 0;
  const int overlap = s - (T - w) > 0 ? s - (T - w) : 0;
  return s + w - overlap;
}

mkv_status cuda_status(cudaError_t e) { return e == cudaSuccess ? MKV_OK : MKV_ERR_CUDA; }

}  // namespace

extern "C" {

const char* mkv_status_str(mkv_status s) {
  switch (s) {
    case MKV_OK: return "ok";
    case MKV_ERR_INVALID_ARG: return "invalid argument";
    case MKV_ERR_SHAPE: return "unsupported or inconsistent shape";
    case MKV_ERR_CAPACITY: return "cache capacity exceeded";
    case MKV_ERR_CUDA: return "CUDA runtime error";
    case MKV_ERR_TIMEOUT: return "device-side wait timed out";
    case MKV_ERR_UNSUPPORTED: return "unsupported head_dim or group";
    case MKV_ERR_WORKSPACE: return "workspace missing, too small or misaligned";
  }
  return "unknown status";
}

int32_t mkv_version(void) { return 202; }

// ------------------------------------------------------------------ decode
size_t mkv_decode_workspace_size(mkv_geom geom, int32_t capacity) {
  if (!geom_ok(geom) || capacity < 1) return 0;
  return decode_workspace_bytes(geom, capacity, num_sms_current());
}

mkv_status mkv_decode_step(mkv_geom geom, const void* q, const void* k_new, const void* v_new,
                           const mkv_cache* cache, const mkv_moments* mom, const mkv_decode_params* p,
                           float* out, float* lse, void* workspace, size_t workspace_bytes, void* stream) {
  NvtxRange nvtx("mkv_decode_step");
  const mkv_status chk = decode_args_status(geom, q, k_new, v_new, cache, mom, p, out);
  if (chk != MKV_OK) return chk;
  const int sms = num_sms_current();
  const size_t need = decode_workspace_bytes(geom, cache->capacity, sms);
  if (!workspace || workspace_bytes < need || !aligned(workspace, 256)) return MKV_ERR_WORKSPACE;
  DecodeArgs a{};
  a.q = q;
  a.k_new = k_new;
  a.v_new = v_new;
  a.K = cache->K;
  a.V = cache->V;
  a.pos = cache->pos;
  a.len = cache->len;
  a.seen = cache->seen;
  a.cap = cache->capacity;
  a.n = p->correction ? mom->n : nullptr;
  a.mu_k = p->correction ? mom->mu_k : nullptr;
  a.mu_v = p->correction ? mom->mu_v : nullptr;
  a.C = p->correction ? mom->C : nullptr;
  a.C16 = p->correction ? static_cast<const __nv_bfloat16*>(p->C16) : nullptr;
  a.Cs = p->correction ? static_cast<const uint2*>(p->C_split) : nullptr;
  a.correction = p->correction;
  a.order = p->order;
  a.tau = p->tau;
  a.out = out;
  a.lse = lse;
  a.batch = geom.batch;
  a.n_kv = geom.n_kv_heads;
  a.early = p->early_load;
  decode_carve(a, geom, cache->capacity, sms, workspace);
  return cuda_status(launch_decode(a, geom.head_dim, geom.group, static_cast<cudaStream_t>(stream)));
}

mkv_status mkv_moments_pack_split(mkv_geom geom, const mkv_moments* mom, float tau, void* C_split, void* stream) {
  NvtxRange nvtx("mkv_moments_pack_split");
  if (!geom_ok(geom)) return geom_status(geom);
  if (!moments_ok(mom) || !C_split || !aligned(C_split, 16) || !(tau >= 0.f)) return MKV_ERR_INVALID_ARG;
  return cuda_status(launch_pack_split(mom->C, mom->n, tau, static_cast<uint2*>(C_split),
                                       geom.batch * geom.n_kv_heads, geom.head_dim, static_cast<cudaStream_t>(stream)));
}

mkv_status mkv_moments_pack_bf16(mkv_geom geom, const mkv_moments* mom, void* C16, void* stream) {
  NvtxRange nvtx("mkv_moments_pack_bf16");
  if (!geom_ok(geom)) return geom_status(geom);
  if (!moments_ok(mom) || !C16 || !aligned(C16, 16)) return MKV_ERR_INVALID_ARG;
  const size_t n = (size_t)geom.batch * geom.n_kv_heads * geom.head_dim * geom.head_dim;
  return cuda_status(launch_pack_bf16(mom->C, static_cast<__nv_bfloat16*>(C16), n, static_cast<cudaStream_t>(stream)));
}

// ------------------------------------------------------------------- evict
size_t mkv_evict_workspace_size(mkv_geom geom, int32_t capacity) {
  if (!geom_ok(geom) || capacity < 1 || capacity > 65536) return 0;
  return evict_workspace_bytes(geom, capacity);
}

mkv_status mkv_evict_append(mkv_geom geom, const void* q, const void* k_new, const void* v_new, int32_t budget,
                            const mkv_cache* cache, const mkv_moments* mom, float tau, void* workspace,
                            size_t workspace_bytes, void* stream) {
  NvtxRange nvtx("mkv_evict_append");
  if (!geom_ok(geom)) return geom_status(geom);
  if (!q || !cache_ok(cache) || !moments_ok(mom) || budget < 0 || !(tau >= 0.f)) return MKV_ERR_INVALID_ARG;
  if ((k_new == nullptr) != (v_new == nullptr)) return MKV_ERR_INVALID_ARG;
  if (cache->capacity > 65536) return MKV_ERR_SHAPE;
  const size_t need = evict_workspace_bytes(geom, cache->capacity);
  if (!workspace || workspace_bytes < need || !aligned(workspace, 256)) return MKV_ERR_WORKSPACE;
  EvictArgs a{};
  a.q = q;
  a.k_new = k_new;
  a.v_new = v_new;
  a.K = cache->K;
  a.V = cache->V;
  a.pos = cache->pos;
  a.len = cache->len;
  a.seen = cache->seen;
  a.cap = cache->capacity;
  a.n = mom->n;
  a.mu_k = mom->mu_k;
  a.mu_v = mom->mu_v;
  a.C = mom->C;
  a.Y = cache->y;
  a.y_len = cache->y_len;
  a.budget = budget;
  a.tau = tau;
  a.batch = geom.batch;
  a.n_kv = geom.n_kv_heads;
  evict_carve(a, geom, cache->capacity, workspace);
  return cuda_status(launch_evict(a, geom.head_dim, geom.group, static_cast<cudaStream_t>(stream)));
}

// ---------------------------------------------------------- decode + evict
// One workspace for both phases: [error header][eviction scratch][decode
// scratch], the decode part carved after the eviction part and both
// reporting into the common header.
static size_t decode_evict_bytes(const mkv_geom& geom, int32_t capacity, int sms) {
  return evict_workspace_bytes(geom, capacity) + decode_workspace_bytes(geom, capacity, sms) - kHeaderBytes;
}

size_t mkv_decode_evict_workspace_size(mkv_geom geom, int32_t capacity) {
  if (!geom_ok(geom) || capacity < 1 || capacity > 65536) return 0;
  return decode_evict_bytes(geom, capacity, num_sms_current());
}

mkv_status mkv_decode_evict_step(mkv_geom geom, const void* q, const void* k_new, const void* v_new, int32_t budget,
                                 const mkv_cache* cache, const mkv_moments* mom, const mkv_decode_params* p,
                                 float* out, float* lse, void* workspace, size_t workspace_bytes, void* stream) {
  NvtxRange nvtx("mkv_decode_evict_step");
  if (!geom_ok(geom)) return geom_status(geom);
  if (!q || !k_new || !v_new || !out || !p || !cache_ok(cache) || !moments_ok(mom) || budget < 0)
    return MKV_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(out, 16) || !aligned(k_new, 16) || !aligned(v_new, 16)) return MKV_ERR_INVALID_ARG;
  if ((p->correction != 0 && p->correction != 1) || (p->order != 0 && p->order != 1) || !(p->tau >= 0.f) ||
      p->C16 != nullptr || p->C_split != nullptr || (p->early_load != 0 && p->early_load != 1))
    return MKV_ERR_INVALID_ARG;
  if (cache->capacity > 65536) return MKV_ERR_SHAPE;
  const int sms = num_sms_current();
  const size_t need = decode_evict_bytes(geom, cache->capacity, sms);
  if (!workspace || workspace_bytes < need || !aligned(workspace, 256)) return MKV_ERR_WORKSPACE;
  EvictArgs e{};
  e.q = q;
  e.k_new = k_new;
  e.v_new = v_new;
  e.K = cache->K;
  e.V = cache->V;
  e.pos = cache->pos;
  e.len = cache->len;
  e.seen = cache->seen;
  e.cap = cache->capacity;
  e.n = mom->n;
  e.mu_k = mom->mu_k;
  e.mu_v = mom->mu_v;
  e.C = mom->C;
  e.Y = cache->y;
  e.y_len = cache->y_len;
  e.budget = budget;
  e.tau = p->tau;
  e.batch = geom.batch;
  e.n_kv = geom.n_kv_heads;
  evict_carve(e, geom, cache->capacity, workspace);
  // Phase 1 by the eviction kernel, then Phase 2 by the decode kernel (whose
  // set-up overlaps the eviction's tail through programmatic dependent launch)
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  cudaError_t ce = launch_evict(e, geom.head_dim, geom.group, st);
  if (ce != cudaSuccess) return cuda_status(ce);
  DecodeArgs a{};
  a.q = q;
  a.K = cache->K;
  a.V = cache->V;
  a.pos = cache->pos;
  a.len = cache->len;
  a.seen = cache->seen;
  a.cap = cache->capacity;
  a.n = p->correction ? mom->n : nullptr;
  a.mu_k = p->correction ? mom->mu_k : nullptr;
  a.mu_v = p->correction ? mom->mu_v : nullptr;
  a.C = p->correction ? mom->C : nullptr;
  a.correction = p->correction;
  a.order = p->order;
  a.tau = p->tau;
  a.out = out;
  a.lse = lse;
  a.batch = geom.batch;
  a.n_kv = geom.n_kv_heads;
  uint8_t* w = static_cast<uint8_t*>(workspace);
  decode_carve(a, geom, cache->capacity, sms, w + evict_workspace_bytes(geom, cache->capacity) - kHeaderBytes);
  a.ws = workspace;
  return cuda_status(launch_decode(a, geom.head_dim, geom.group, st));
}

// ---------------------------------------------------------------- compress
static mkv_status compress_params_ok(const mkv_geom& geom, int32_t T, const mkv_compress_params* p) {
  if (!geom_ok(geom)) return geom_status(geom);
  if (!p || T < 1 || T > (1 << 20) || p->budget < 1 || p->window < 1 || p->window > T || p->sink < 0)
    return MKV_ERR_INVALID_ARG;
  if ((p->keep_window != 0 && p->keep_window != 1) || (p->mi != 0 && p->mi != 1) ||
      (p->causal != 0 && p->causal != 1) || !(p->tau >= 0.f))
    return MKV_ERR_INVALID_ARG;
  if (!(p->pool == 1 || p->pool == 2 || p->pool == 4 || p->pool == 8 || p->pool == 16 || p->pool == 32))
    return MKV_ERR_INVALID_ARG;
  // the g * w window rows fill at most two 128-row blocks: the Q stage in
  // shared memory, the logits columns in TMEM and one Q tensor-map box
  if ((long)geom.group * p->window > 256) return MKV_ERR_SHAPE;
  // the compress kernels take one grid row (y) per unit
  if ((long)geom.batch * geom.n_kv_heads > 65535) return MKV_ERR_SHAPE;
  if (T > p->budget && protected_count_host(T, p->window, p->sink, p->keep_window) > p->budget)
    return MKV_ERR_INVALID_ARG;
  if (p->adaptive != 0 && p->adaptive != 1) return MKV_ERR_INVALID_ARG;
  if (p->adaptive && (geom.n_kv_heads > 64 || (long)geom.n_kv_heads * T > (1L << 28))) return MKV_ERR_SHAPE;
  return MKV_OK;
}

// rows one unit may retain: min(T, budget), or with the adaptive allocation
// the unit's protected rows plus every joint selection of its batch item
static long max_retained(const mkv_geom& geom, int32_t T, const mkv_compress_params* p) {
  if (T <= p->budget || !p->adaptive) return T < p->budget ? T : p->budget;
  const long prot = protected_count_host(T, p->window, p->sink, p->keep_window);
  const long m = (long)geom.n_kv_heads * (p->budget - prot) + prot;
  return m < T ? m : T;
}

size_t mkv_compress_workspace_size(mkv_geom geom, int32_t T, const mkv_compress_params* p) {
  if (compress_params_ok(geom, T, p) != MKV_OK) return 0;
  return compress_workspace_bytes(geom, T, *p, num_sms_current());
}

mkv_status mkv_compress(mkv_geom geom, int32_t T, const void* K, const void* V, const void* Q_obs,
                        const mkv_compress_params* p, const mkv_cache* out_cache, const mkv_moments* out_mom,
                        const mkv_compress_diag* diag, void* workspace, size_t workspace_bytes, void* stream) {
  NvtxRange nvtx("mkv_compress");
  mkv_status st = compress_params_ok(geom, T, p);
  if (st != MKV_OK) return st;
  if (!K || !V || !Q_obs || !cache_ok(out_cache) || !moments_ok(out_mom)) return MKV_ERR_INVALID_ARG;
  if (!aligned(K, 16) || !aligned(V, 16) || !aligned(Q_obs, 16)) return MKV_ERR_INVALID_ARG;
  if (out_cache->capacity < max_retained(geom, T, p)) return MKV_ERR_CAPACITY;
  const int sms = num_sms_current();
  const size_t need = compress_workspace_bytes(geom, T, *p, sms);
  if (!workspace || workspace_bytes < need || !aligned(workspace, 256)) return MKV_ERR_WORKSPACE;
  CompressArgs a{};
  a.K = K;
  a.V = V;
  a.Q = Q_obs;
  a.T = T;
  a.budget = p->budget;
  a.window = p->window;
  a.sink = p->sink;
  a.keep_window = p->keep_window;
  a.pool = p->pool;
  a.mi = p->mi;
  a.causal = p->causal;
  a.tau = p->tau;
  a.adaptive = p->adaptive;
  a.cache = *out_cache;
  a.mom = *out_mom;
  a.diag_scores = diag ? diag->scores : nullptr;
  a.diag_score2 = diag ? diag->score2 : nullptr;
  a.diag_idx1 = diag ? diag->idx_stage1 : nullptr;
  a.ws = workspace;
  a.batch = geom.batch;
  a.n_kv = geom.n_kv_heads;
  // the cache's rows and the moments are replaced: no y row stays current
  if (out_cache->y_len != nullptr &&
      cudaMemsetAsync(out_cache->y_len, 0, (size_t)geom.batch * geom.n_kv_heads * sizeof(int32_t),
                      static_cast<cudaStream_t>(stream)) != cudaSuccess)
    return MKV_ERR_CUDA;
  return cuda_status(launch_compress(a, geom, workspace_bytes, sms, static_cast<cudaStream_t>(stream)));
}

// ------------------------------------------------------------- test hooks
int64_t mkv_debug_set_poll_limit(int64_t polls) {
  const uint32_t v = polls < 0 ? kMaxPolls : (polls > (int64_t)kMaxPolls ? kMaxPolls : static_cast<uint32_t>(polls));
  return static_cast<int64_t>(g_poll_limit.exchange(v));
}

int32_t mkv_debug_force_ticket_merge(int32_t on) { return g_force_ticket_merge.exchange(on != 0 ? 1 : 0); }

// ------------------------------------------------------------------ errors
mkv_status mkv_get_device_error(void* workspace, void* stream, int32_t* info) {
  if (!workspace) return MKV_ERR_WORKSPACE;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  ErrorWord w{};
  if (cudaMemcpyAsync(&w, workspace, sizeof(w), cudaMemcpyDeviceToHost, s) != cudaSuccess) return MKV_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return MKV_ERR_CUDA;
  if (w.code != 0) {
    if (cudaMemsetAsync(workspace, 0, sizeof(w), s) != cudaSuccess) return MKV_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return MKV_ERR_CUDA;
  }
  if (info) *info = w.info;
  return static_cast<mkv_status>(w.code);
}

}  // extern "C"
