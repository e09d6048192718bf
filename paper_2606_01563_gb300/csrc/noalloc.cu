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
// loads this library keeps until the process exits.  The error word at its
// start is never cleared: the first error a kernel records stays set for the
// life of the process (this entry point has no workspace to read it from).
#include <cuda_runtime.h>

#include <mutex>

#include "common.cuh"
#include "kernels.h"
#include "validate.h"

using namespace mkv;

namespace {

constexpr size_t kNoAllocScratchBytes = size_t(4) << 20;  // 4 MiB per device
// Ticket counters sit in a region of their own at a fixed offset, sized for
// the most units any accepted geometry has (each unit needs at least 528
// bytes of partial records, so fewer than 8192 units fit in 4 MiB).  Partial
// records of one call therefore never land where another call's counters
// are; each merge returns its counter to zero.
constexpr size_t kMaxUnits = 8192;
constexpr size_t kCounterBytes = kMaxUnits * sizeof(uint32_t);
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_decode_scratch[kNoAllocScratchBytes];

std::mutex g_setup_mutex;
void* g_scratch_ptr[kMaxDevices] = {nullptr};
int g_num_sms[kMaxDevices] = {0};

// Every call, with the device current: look up the array's device address
// (its name in host code is only a stand-in).  The first time a device is
// seen, or when the address changed (the module was loaded again, e.g. after
// cudaDeviceReset), zero the array so that the error word and the ticket
// counters start at zero; that set-up synchronises the device.
mkv_status setup_current_device(void** scratch, int* sms) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return MKV_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return MKV_ERR_UNSUPPORTED;
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_decode_scratch) != cudaSuccess || p == nullptr) return MKV_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  if (g_scratch_ptr[dev] != p) {
    if (cudaMemset(p, 0, kNoAllocScratchBytes) != cudaSuccess) return MKV_ERR_CUDA;
    if (cudaDeviceSynchronize() != cudaSuccess) return MKV_ERR_CUDA;
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
    g_num_sms[dev] = n;
    g_scratch_ptr[dev] = p;
  }
  *scratch = p;
  *sms = g_num_sms[dev];
  return MKV_OK;
}

// Bytes of the array a call with S splits per unit uses:
// [error header][counters, fixed][partials][f_hat_E rows].
size_t scratch_bytes(const mkv_geom& g, int S) {
  const size_t units = (size_t)g.batch * g.n_kv_heads;
  return kHeaderBytes + kCounterBytes + align_up(units * S * g.group * (g.head_dim + 4) * sizeof(float), 256) +
         align_up(units * g.group * g.head_dim * sizeof(float), 256);
}

void carve(DecodeArgs& a, const mkv_geom& g, int S, int sms, void* scratch) {
  const size_t units = (size_t)g.batch * g.n_kv_heads;
  uint8_t* p = static_cast<uint8_t*>(scratch);
  a.ws = scratch;
  a.counters = reinterpret_cast<uint32_t*>(p + kHeaderBytes);
  a.partial = reinterpret_cast<float*>(p + kHeaderBytes + kCounterBytes);
  a.fhat = reinterpret_cast<float*>(p + kHeaderBytes + kCounterBytes +
                                    align_up(units * S * g.group * (g.head_dim + 4) * sizeof(float), 256));
  a.S = S;
  a.S_cl = decode_cluster_splits(g, a.cap, sms, a.early);
}

}  // namespace

extern "C" MKV_API mkv_status mkv_decode_step_noalloc(mkv_geom geom, const void* q, const void* k_new,
                                                      const void* v_new, const mkv_cache* cache,
                                                      const mkv_moments* mom, const mkv_decode_params* p,
                                                      float* out, float* lse, void* stream) {
  NvtxRange nvtx("mkv_decode_step_noalloc");
  const mkv_status chk = decode_args_status(geom, q, k_new, v_new, cache, mom, p, out);
  if (chk != MKV_OK) return chk;
  // The smallest split count needs one partial record per query head: reject
  // geometries whose scratch would exceed the fixed array before any set-up.
  if ((size_t)geom.batch * geom.n_kv_heads > kMaxUnits || scratch_bytes(geom, 1) > kNoAllocScratchBytes)
    return MKV_ERR_WORKSPACE;

  void* scratch = nullptr;
  int sms = 0;
  mkv_status st = setup_current_device(&scratch, &sms);
  if (st != MKV_OK) return st;
  int S = decode_splits(geom, cache->capacity, sms);
  while (S > 1 && scratch_bytes(geom, S) > kNoAllocScratchBytes) --S;

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
  carve(a, geom, S, sms, scratch);
  return launch_decode(a, geom.head_dim, geom.group, static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? MKV_OK
             : MKV_ERR_CUDA;
}
