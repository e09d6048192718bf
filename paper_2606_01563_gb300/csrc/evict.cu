// Moment-informed eviction (Algorithm 1: append step and Phase 1).
//
// One CTA per unit runs the eviction loop literally: every iteration
// recomputes alpha (softmax over the surviving rows, summed over the G query
// heads of the unit) and every surviving row's moment residual
//   r_j = v_j - v_bar - scale * C' k_j,  C' = C with |n C_ab| < tau zeroed
// (Eq. residual with S_tilde = n C), evicts the argmin of alpha_j ||r_j||
// (ties: lower row = lower position), and folds the evicted row into
// (n, mu_k, mu_v, C) with the Welford form of Eq. app_update.  C lives in
// shared memory transposed (Ct[c][a] = C[a][c]) so that a warp's lanes read
// consecutive output dims of one column: conflict-free 128-bit loads while
// the key element is a broadcast.  Rows are compacted in order at the end.
#include "common.cuh"
#include "kernels.h"

namespace mkv {

namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kRowsPerGroup = 4;  // rows a warp scores together
constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ unsigned long long shfl_min_u64(unsigned long long v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long w = __shfl_xor_sync(kFull, v, o);
    v = w < v ? w : v;
  }
  return v;
}

template <int D, int G>
__global__ void __launch_bounds__(kThreads) evict_kernel(const EvictArgs a) {
  constexpr int DPL = D / 32;
  extern __shared__ __align__(16) uint8_t dsmem[];
  float* Ct = reinterpret_cast<float*>(dsmem);                        // [D][D] transposed C
  float* kbuf = Ct + D * D;                                           // [warps][4][D]
  uint8_t* alive = reinterpret_cast<uint8_t*>(kbuf + kWarps * kRowsPerGroup * D);  // [cap]
  __shared__ float s_mu_k[D], s_mu_v[D], s_dk[D], s_dv[D];
  __shared__ float s_q[G][D];  // q * scale
  __shared__ float s_m[G], s_z[G];
  __shared__ float s_red[kWarps][G];
  __shared__ unsigned long long s_best[kWarps];
  __shared__ int s_jstar;

  const int u = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int len_in = a.len[u];
  const bool has_new = a.k_new != nullptr;
  const size_t row0 = (size_t)u * a.cap;
  __nv_bfloat16* Kg = reinterpret_cast<__nv_bfloat16*>(a.K) + row0 * D;
  __nv_bfloat16* Vg = reinterpret_cast<__nv_bfloat16*>(a.V) + row0 * D;
  int32_t* Pg = a.pos + row0;

  if (len_in < 0 || len_in > a.cap || (has_new && len_in + 1 > a.cap)) {
    if (tid == 0) record_error(a.ws, MKV_ERR_CAPACITY, u);
    return;
  }
  if (has_new) {
    const __nv_bfloat16* kn = reinterpret_cast<const __nv_bfloat16*>(a.k_new) + (size_t)u * D;
    const __nv_bfloat16* vn = reinterpret_cast<const __nv_bfloat16*>(a.v_new) + (size_t)u * D;
    for (int i = tid; i < D; i += kThreads) {
      Kg[(size_t)len_in * D + i] = kn[i];
      Vg[(size_t)len_in * D + i] = vn[i];
    }
    if (tid == 0) {
      Pg[len_in] = a.seen[u];
      a.seen[u] = a.seen[u] + 1;
    }
  }
  const int len = len_in + (has_new ? 1 : 0);
  if (len <= a.budget) {
    if (tid == 0) a.len[u] = len;
    return;
  }

  int n = a.n[u];
  for (int idx = tid; idx < D * D; idx += kThreads) {
    const int r = idx / D, c = idx % D;
    Ct[c * D + r] = (n > 0) ? a.C[(size_t)u * D * D + idx] : 0.f;
  }
  for (int i = tid; i < D; i += kThreads) {
    s_mu_k[i] = (n > 0) ? a.mu_k[(size_t)u * D + i] : 0.f;
    s_mu_v[i] = (n > 0) ? a.mu_v[(size_t)u * D + i] : 0.f;
  }
  const float scale = rsqrtf(static_cast<float>(D));
  const __nv_bfloat16* qg = reinterpret_cast<const __nv_bfloat16*>(a.q) + (size_t)u * G * D;
  for (int i = tid; i < G * D; i += kThreads) s_q[i / D][i % D] = __bfloat162float(qg[i]) * scale;
  for (int j = tid; j < len; j += kThreads) alive[j] = 1;
  __syncthreads();

  // logits lg[h][j] = scale q_h . k_j (fixed for the whole call)
  float* lg = a.scratch + (size_t)u * G * a.cap;
  for (int j = warp; j < len; j += kWarps) {
    float kf[DPL];
    load_bf16<DPL>(Kg + (size_t)j * D + lane * DPL, kf);
#pragma unroll
    for (int h = 0; h < G; ++h) {
      float acc = 0.f;
#pragma unroll
      for (int i = 0; i < DPL; ++i) acc = fmaf(s_q[h][lane * DPL + i], kf[i], acc);
      acc = warp_sum(acc);
      if (lane == 0) lg[(size_t)h * a.cap + j] = acc;
    }
  }
  __syncthreads();

  const int n_evict = len - a.budget;
  const float tau = a.tau;
  for (int e = 0; e < n_evict; ++e) {
    // ---- per-head softmax normaliser over the surviving rows
    {
      float mx[G];
#pragma unroll
      for (int h = 0; h < G; ++h) mx[h] = -INFINITY;
      for (int j = tid; j < len; j += kThreads)
        if (alive[j]) {
#pragma unroll
          for (int h = 0; h < G; ++h) mx[h] = fmaxf(mx[h], lg[(size_t)h * a.cap + j]);
        }
#pragma unroll
      for (int h = 0; h < G; ++h) {
        mx[h] = warp_max(mx[h]);
        if (lane == 0) s_red[warp][h] = mx[h];
      }
      __syncthreads();
      if (tid < G) {
        float m = -INFINITY;
        for (int w = 0; w < kWarps; ++w) m = fmaxf(m, s_red[w][tid]);
        s_m[tid] = m;
      }
      __syncthreads();
      float zs[G];
#pragma unroll
      for (int h = 0; h < G; ++h) zs[h] = 0.f;
      for (int j = tid; j < len; j += kThreads)
        if (alive[j]) {
#pragma unroll
          for (int h = 0; h < G; ++h) zs[h] += expf(lg[(size_t)h * a.cap + j] - s_m[h]);
        }
#pragma unroll
      for (int h = 0; h < G; ++h) {
        zs[h] = warp_sum(zs[h]);
        if (lane == 0) s_red[warp][h] = zs[h];
      }
      __syncthreads();
      if (tid < G) {
        float z = 0.f;
        for (int w = 0; w < kWarps; ++w) z += s_red[w][tid];
        s_z[tid] = z;
      }
      __syncthreads();
    }

    // ---- scores of the surviving rows, groups of 4 rows per warp
    const float nf = static_cast<float>(n);
    const float rs = (n > 0) ? scale : 0.f;
    unsigned long long best = ~0ull;
    float* kb = kbuf + warp * kRowsPerGroup * D;
    for (int g0 = warp * kRowsPerGroup; g0 < len; g0 += kWarps * kRowsPerGroup) {
      bool any = false;
#pragma unroll
      for (int r = 0; r < kRowsPerGroup; ++r) any |= (g0 + r < len) && alive[g0 + r];
      if (!any) continue;  // warp-uniform
#pragma unroll
      for (int r = 0; r < kRowsPerGroup; ++r) {
        float kf[DPL];
        if (g0 + r < len) {
          load_bf16<DPL>(Kg + (size_t)(g0 + r) * D + lane * DPL, kf);
        } else {
#pragma unroll
          for (int i = 0; i < DPL; ++i) kf[i] = 0.f;
        }
#pragma unroll
        for (int i = 0; i < DPL; ++i) kb[r * D + lane * DPL + i] = kf[i];
      }
      __syncwarp();
      float y[kRowsPerGroup][DPL];
#pragma unroll
      for (int r = 0; r < kRowsPerGroup; ++r)
#pragma unroll
        for (int i = 0; i < DPL; ++i) y[r][i] = 0.f;
      if (n > 0) {
#pragma unroll 4
        for (int c = 0; c < D; ++c) {
          float cv[DPL];
          if constexpr (DPL == 4) {
            const float4 t = *reinterpret_cast<const float4*>(Ct + c * D + lane * 4);
            cv[0] = t.x; cv[1] = t.y; cv[2] = t.z; cv[3] = t.w;
          } else {
            const float2 t = *reinterpret_cast<const float2*>(Ct + c * D + lane * 2);
            cv[0] = t.x; cv[1] = t.y;
          }
#pragma unroll
          for (int i = 0; i < DPL; ++i) cv[i] = (fabsf(cv[i] * nf) < tau) ? 0.f : cv[i];
#pragma unroll
          for (int r = 0; r < kRowsPerGroup; ++r) {
            const float kc = kb[r * D + c];
#pragma unroll
            for (int i = 0; i < DPL; ++i) y[r][i] = fmaf(cv[i], kc, y[r][i]);
          }
        }
      }
#pragma unroll
      for (int r = 0; r < kRowsPerGroup; ++r) {
        const int j = g0 + r;
        const bool live = (j < len) && alive[j];
        float vf[DPL];
        if (live) {
          load_bf16<DPL>(Vg + (size_t)j * D + lane * DPL, vf);
        } else {
#pragma unroll
          for (int i = 0; i < DPL; ++i) vf[i] = 0.f;
        }
        float ss = 0.f;
#pragma unroll
        for (int i = 0; i < DPL; ++i) {
          const float rr = vf[i] - s_mu_v[lane * DPL + i] - rs * y[r][i];
          ss = fmaf(rr, rr, ss);
        }
        ss = warp_sum(ss);
        if (live) {
          float alpha = 0.f;
#pragma unroll
          for (int h = 0; h < G; ++h) alpha += expf(lg[(size_t)h * a.cap + j] - s_m[h]) / s_z[h];
          const float score = alpha * sqrtf(ss);
          const unsigned long long key =
              (static_cast<unsigned long long>(__float_as_uint(score)) << 32) | static_cast<unsigned>(j);
          best = key < best ? key : best;
        }
      }
      __syncwarp();
    }
    best = shfl_min_u64(best);
    if (lane == 0) s_best[warp] = best;
    __syncthreads();
    if (tid == 0) {
      unsigned long long b = s_best[0];
      for (int w = 1; w < kWarps; ++w) b = s_best[w] < b ? s_best[w] : b;
      const int js = static_cast<int>(b & 0xffffffffu);
      s_jstar = js;
      alive[js] = 0;
    }
    __syncthreads();

    // ---- fold row j* into the moments (Welford form of Eq. app_update)
    const int js = s_jstar;
    const float n1 = static_cast<float>(n + 1);
    for (int i = tid; i < D; i += kThreads) {
      const float kx = __bfloat162float(Kg[(size_t)js * D + i]);
      const float vx = __bfloat162float(Vg[(size_t)js * D + i]);
      const float dk = kx - s_mu_k[i];
      s_mu_k[i] += dk / n1;
      const float mv = s_mu_v[i] + (vx - s_mu_v[i]) / n1;
      s_mu_v[i] = mv;
      s_dk[i] = dk;
      s_dv[i] = vx - mv;
    }
    __syncthreads();
    const float keep = static_cast<float>(n) / n1;
    const float inv = 1.f / n1;
    for (int idx = tid; idx < D * D; idx += kThreads) {
      const int c = idx / D, r = idx % D;  // Ct[c][r] = C[r][c]
      Ct[idx] = keep * Ct[idx] + inv * s_dv[r] * s_dk[c];
    }
    n += 1;
    __syncthreads();
  }

  // ---- write the moments back
  for (int idx = tid; idx < D * D; idx += kThreads) {
    const int r = idx / D, c = idx % D;
    a.C[(size_t)u * D * D + idx] = Ct[c * D + r];
  }
  for (int i = tid; i < D; i += kThreads) {
    a.mu_k[(size_t)u * D + i] = s_mu_k[i];
    a.mu_v[(size_t)u * D + i] = s_mu_v[i];
  }
  if (tid == 0) {
    a.n[u] = n;
    a.len[u] = a.budget;
  }

  // ---- ordered in-place compaction, 32 rows per step (destination <= source)
  int base = 0;
  for (int c0 = 0; c0 < len; c0 += 32) {
    const bool al = (c0 + lane < len) && alive[c0 + lane];
    const unsigned mask = __ballot_sync(kFull, al);
    // warp w moves rows c0 + 4w .. c0 + 4w + 3
    uint2 kreg[4], vreg[4];
    int32_t preg[4];
    int dst[4];
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int j = c0 + warp * 4 + r;
      const int bit = warp * 4 + r;
      dst[r] = -1;
      if (j < len && ((mask >> bit) & 1u)) {
        dst[r] = base + __popc(mask & ((1u << bit) - 1u));
        if constexpr (DPL == 4) {
          kreg[r] = *reinterpret_cast<const uint2*>(Kg + (size_t)j * D + lane * 4);
          vreg[r] = *reinterpret_cast<const uint2*>(Vg + (size_t)j * D + lane * 4);
        } else {
          kreg[r].x = *reinterpret_cast<const uint32_t*>(Kg + (size_t)j * D + lane * 2);
          vreg[r].x = *reinterpret_cast<const uint32_t*>(Vg + (size_t)j * D + lane * 2);
        }
        preg[r] = Pg[j];
      }
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      if (dst[r] >= 0) {
        if constexpr (DPL == 4) {
          *reinterpret_cast<uint2*>(Kg + (size_t)dst[r] * D + lane * 4) = kreg[r];
          *reinterpret_cast<uint2*>(Vg + (size_t)dst[r] * D + lane * 4) = vreg[r];
        } else {
          *reinterpret_cast<uint32_t*>(Kg + (size_t)dst[r] * D + lane * 2) = kreg[r].x;
          *reinterpret_cast<uint32_t*>(Vg + (size_t)dst[r] * D + lane * 2) = vreg[r].x;
        }
        if (lane == 0) Pg[dst[r]] = preg[r];
      }
    }
    base += __popc(mask);
    __syncthreads();
  }
}

template <int D, int G>
cudaError_t launch_dg(const EvictArgs& a, cudaStream_t stream) {
  const size_t smem = (size_t)D * D * 4 + (size_t)kWarps * kRowsPerGroup * D * 4 + align_up(a.cap, 16);
  cudaError_t e = cudaFuncSetAttribute(evict_kernel<D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  evict_kernel<D, G><<<a.batch * a.n_kv, kThreads, smem, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace

size_t evict_workspace_bytes(const mkv_geom& g, int32_t capacity) {
  const size_t units = (size_t)g.batch * g.n_kv_heads;
  return kHeaderBytes + align_up(units * g.group * (size_t)capacity * sizeof(float), 256);
}

void evict_carve(EvictArgs& a, const mkv_geom& g, int32_t capacity, void* ws) {
  (void)g;
  (void)capacity;
  a.ws = ws;
  a.scratch = reinterpret_cast<float*>(static_cast<uint8_t*>(ws) + kHeaderBytes);
}

cudaError_t launch_evict(const EvictArgs& a, int head_dim, int group, cudaStream_t stream) {
#define MKV_EVICT_CASE(D, G) \
  if (head_dim == D && group == G) return launch_dg<D, G>(a, stream);
  MKV_EVICT_CASE(128, 1)
  MKV_EVICT_CASE(128, 2)
  MKV_EVICT_CASE(128, 4)
  MKV_EVICT_CASE(128, 8)
  MKV_EVICT_CASE(64, 1)
  MKV_EVICT_CASE(64, 2)
  MKV_EVICT_CASE(64, 4)
  MKV_EVICT_CASE(64, 8)
#undef MKV_EVICT_CASE
  return cudaErrorInvalidValue;
}

}  // namespace mkv
