// Shared device helpers for the MomentKV kernels (sm_103a).
//
// Every workspace starts with a 256-byte header holding the device error
// word: [0] status code (first error wins), [1] detail word.  Kernels record
// into it instead of trapping; mkv_get_device_error reads and clears it.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>
#include <stdint.h>

#include <atomic>
#include <mutex>

#include "../../include/mkv.h"

namespace mkv {

constexpr size_t kHeaderBytes = 256;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
// Upper bound on polls of one mbarrier phase before a wait gives up.  Each
// poll is a try_wait that may itself suspend for a while, so this is well
// over a second -- far beyond any legitimate copy latency.
constexpr uint32_t kMaxPolls = 1u << 22;

// Poll limit of the pipeline waits (tile copies, MMA commits), passed to the
// kernels in their arguments.  Normally kMaxPolls; mkv_debug_set_poll_limit
// lowers it so that a test can make those waits run out.  The waits that
// drain a CTA's copies in flight before it exits always use kMaxPolls.
inline std::atomic<uint32_t> g_poll_limit{kMaxPolls};
inline uint32_t pipeline_poll_limit() { return g_poll_limit.load(std::memory_order_relaxed); }
// Test switch: the decode merges through global partial records (the variant
// that runs when a cluster of the split count cannot be co-scheduled).
inline std::atomic<int> g_force_ticket_merge{0};

struct ErrorWord {
  uint32_t code;
  int32_t info;
};

__device__ __forceinline__ void record_error(void* ws, uint32_t code, int32_t info) {
  ErrorWord* e = reinterpret_cast<ErrorWord*>(ws);
  if (atomicCAS(&e->code, 0u, code) == 0u) {
    atomicExch(reinterpret_cast<int*>(&e->info), info);
  }
}

__host__ __device__ __forceinline__ size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// ---------------------------------------------------------------- mbarrier
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_fence_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_addr(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait on one phase (at most `polls` polls); returns false if it gave up.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, uint32_t polls = kMaxPolls) {
  for (uint32_t i = 0; i < polls; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
  }
  return false;
}

// ------------------------------------------------------- bulk async copies
// 1-D bulk copy global -> shared completing on an mbarrier (TMA engine).
// dst, src 16-byte aligned; bytes a multiple of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(bar))
      : "memory");
}

// 2-D tiled bulk copy (TMA) global -> shared through a tensor map; x is the
// inner (element) coordinate and must be a multiple of 16 bytes' worth of
// elements, y the row.  Out-of-range elements are filled with zeros.
__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar))
      : "memory");
}

// L2 eviction-priority policies for cache hints: evict_last for small data
// read again on every call (moments, cache lengths), evict_first for data
// streamed through once per call (cache rows).
__device__ __forceinline__ uint64_t l2_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
// Read-only loads with an L2 cache policy.
__device__ __forceinline__ float ldg_hint(const float* p, uint64_t pol) {
  float v;
  asm volatile("ld.global.nc.L2::cache_hint.f32 %0, [%1], %2;" : "=f"(v) : "l"(p), "l"(pol));
  return v;
}
__device__ __forceinline__ float2 ldg_hint(const float2* p, uint64_t pol) {
  float2 v;
  asm volatile("ld.global.nc.L2::cache_hint.v2.f32 {%0, %1}, [%2], %3;" : "=f"(v.x), "=f"(v.y) : "l"(p), "l"(pol));
  return v;
}
__device__ __forceinline__ uint32_t ldg_hint(const uint32_t* p, uint64_t pol) {
  uint32_t v;
  asm volatile("ld.global.nc.L2::cache_hint.b32 %0, [%1], %2;" : "=r"(v) : "l"(p), "l"(pol));
  return v;
}
// A coherent (L2) load and a store of an int32 with an L2 cache policy.
__device__ __forceinline__ int32_t ldcg_hint(const int32_t* p, uint64_t pol) {
  int32_t v;
  asm volatile("ld.global.cg.L2::cache_hint.s32 %0, [%1], %2;" : "=r"(v) : "l"(p), "l"(pol) : "memory");
  return v;
}
__device__ __forceinline__ void st_hint(int32_t* p, int32_t v, uint64_t pol) {
  asm volatile("st.global.L2::cache_hint.s32 [%0], %1, %2;" ::"l"(p), "r"(v), "l"(pol) : "memory");
}

// tma_load_2d with an L2 cache policy on the bytes it reads.
__device__ __forceinline__ void tma_load_2d_hint(void* dst, const CUtensorMap* map, int x, int y, uint64_t* bar,
                                                 uint64_t pol) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%2, "
      "%3}], [%4], %5;" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar)), "l"(pol)
      : "memory");
}

// Host: encode a row-major bf16 matrix [rows][inner] (row stride in bytes) as a
// 2-D tensor map with a box of box_rows x box_inner elements and the 128-byte
// swizzle (box_inner * 2 <= 128).  Returns false if the driver refuses it.
inline bool encode_tmap_bf16(CUtensorMap* map, const void* base, uint64_t inner, uint64_t rows,
                             uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_rows) {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  if (fn == nullptr) return false;
  const cuuint64_t dims[2] = {inner, rows};
  const cuuint64_t strides[1] = {row_stride_bytes};
  const cuuint32_t box[2] = {box_inner, box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Byte offset of element (r, c) in a tile of `rows` rows stored as boxes of 64
// bf16 columns (128 B per row) with the 128-byte swizzle: within each 8-row
// group, the 16-byte chunk index is XORed with (row mod 8).
__device__ __forceinline__ uint32_t swz_off(int r, int c, int rows) {
  const int box = c >> 6, cc = c & 63;
  return static_cast<uint32_t>(box * rows * 128 + r * 128 + ((((cc >> 3) ^ (r & 7))) << 4) + (cc & 7) * 2);
}

// ----------------------------------------------------------------- numeric
// 2^x on the special-function unit (relative error ~2^-22; results below
// 2^-126 flush to 0, which only ever drops negligible softmax weights).
__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Order-preserving map of a float to uint32 (larger float -> larger key).
__device__ __forceinline__ uint32_t float_key(float f) {
  uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// Load N consecutive bf16 as floats (N in {2, 4, 8}); p must be aligned to 2N bytes.
template <int N>
__device__ __forceinline__ void load_bf16(const __nv_bfloat16* p, float* out) {
  if constexpr (N == 2) {
    __nv_bfloat162 v = *reinterpret_cast<const __nv_bfloat162*>(p);
    out[0] = __low2float(v);
    out[1] = __high2float(v);
  } else if constexpr (N == 4) {
    uint2 raw = *reinterpret_cast<const uint2*>(p);
    __nv_bfloat162 a = *reinterpret_cast<__nv_bfloat162*>(&raw.x);
    __nv_bfloat162 b = *reinterpret_cast<__nv_bfloat162*>(&raw.y);
    out[0] = __low2float(a);
    out[1] = __high2float(a);
    out[2] = __low2float(b);
    out[3] = __high2float(b);
  } else {
    uint4 raw = *reinterpret_cast<const uint4*>(p);
    const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      __nv_bfloat162 v = *reinterpret_cast<const __nv_bfloat162*>(&w[i]);
      out[2 * i] = __low2float(v);
      out[2 * i + 1] = __high2float(v);
    }
  }
}

}  // namespace mkv
