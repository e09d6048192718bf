// mkv_decode_step_noalloc: the decode step with its scratch in a fixed
// device array instead of a caller-provided workspace.
//
// Some callers cannot allocate device memory at the point where they decode:
// a plugin inside a host inference engine that hands it only input and output
// buffers, a serving process whose device memory was reserved up front by
// another allocator, or a latency-critical path where cudaMalloc's implicit
// device synchronisation is not acceptable.  For them the split-K partial
// states, ticket counters and moment rows live in `g_decode_scratch` below:
// a file-scope device array of kNoAllocScratchBytes that every GPU which
// loads this library keeps until the process exits.
#include <cuda_runtime.h>

#include <mutex>

#include "common.cuh"
#include "kernels.h"

using namespace mkv;

namespace {

constexpr size_t kNoAllocScratchBytes = size_t(4) << 20;  // 4 MiB per device
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_decode_scratch[kNoAllocScratchBytes];

std::mutex g_setup_mutex;
void* g_scratch_ptr[kMaxDevices] = {nullptr};
int g_num_sms[kMaxDevices] = {0};

// Once per device, with that device current: look up the array's device
// address (its name in host code is only a stand-in) and zero it, so the
// error word and the ticket counters start at zero.  Synchronises the device.
mkv_status setup_current_device(void** scratch, int* sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return MKV_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return MKV_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (g_scratch_ptr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_decode_scratch) != cudaSuccess || p == nullptr) return MKV_ERR_CUDA;
    if (cudaMemset(p, 0, kNoAllocScratchBytes) != cudaSuccess) return MKV_ERR_CUDA;
    if (cudaDeviceSynchronize() != cudaSuccess) return MKV_ERR_CUDA;
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
    g_num_sms[dev] = n;
    g_scratch_ptr[dev] = p;
  }
  *scratch = g_scratch_ptr[dev];
  *sms = g_num_sms[dev];
  return MKV_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) % 16) == 0; }

}  // namespace

extern "C" MKV_API mkv_status mkv_decode_step_noalloc(mkv_geom geom, const void* q, const void* k_new,
                                                      const void* v_new, const mkv_cache* cache,
                                                      const mkv_moments* mom, const mkv_decode_params* p,
                                                      float* out, float* lse, void* stream) {
  const bool dims_ok = geom.head_dim == 64 || geom.head_dim == 128;
  const bool group_ok = geom.group == 1 || geom.group == 2 || geom.group == 4 || geom.group == 8;
  if (!dims_ok) return MKV_ERR_UNSUPPORTED;
  if (!group_ok || geom.batch < 1 || geom.n_kv_heads < 1 || (long)geom.batch * geom.n_kv_heads > 65535L * 64)
    return MKV_ERR_SHAPE;
  if (!q || !out || !p || !cache || !cache->K || !cache->V || !cache->pos || !cache->len || !cache->seen ||
      cache->capacity < 1 || !aligned16(cache->K) || !aligned16(cache->V))
    return MKV_ERR_INVALID_ARG;
  if ((k_new == nullptr) != (v_new == nullptr)) return MKV_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(out) || (k_new && (!aligned16(k_new) || !aligned16(v_new))))
    return MKV_ERR_INVALID_ARG;
  if ((p->correction != 0 && p->correction != 1) || (p->order != 0 && p->order != 1) || !(p->tau >= 0.f))
    return MKV_ERR_INVALID_ARG;
  if (p->correction && (!mom || !mom->n || !mom->mu_k || !mom->mu_v || !mom->C || !aligned16(mom->C)))
    return MKV_ERR_INVALID_ARG;
  if (p->C16 && !aligned16(p->C16)) return MKV_ERR_INVALID_ARG;
  // The smallest split count needs one partial record per query head: reject
  // geometries whose scratch would exceed the fixed array before any set-up.
  if (decode_workspace_bytes_splits(geom, 1) > kNoAllocScratchBytes) return MKV_ERR_WORKSPACE;

  void* scratch = nullptr;
  int sms = 0;
  mkv_status st = setup_current_device(&scratch, &sms);
  if (st != MKV_OK) return st;
  int S = decode_splits(geom, cache->capacity, sms);
  while (S > 1 && decode_workspace_bytes_splits(geom, S) > kNoAllocScratchBytes) --S;

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
  a.correction = p->correction;
  a.order = p->order;
  a.tau = p->tau;
  a.out = out;
  a.lse = lse;
  a.batch = geom.batch;
  a.n_kv = geom.n_kv_heads;
  decode_carve_splits(a, geom, S, scratch);
  return launch_decode(a, geom.head_dim, geom.group, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? MKV_OK
             : MKV_ERR_CUDA;
}
