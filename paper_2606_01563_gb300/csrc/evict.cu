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
//
// Two kernels compute the same thing:
//  - evict_cluster_kernel (used whenever a row slice fits in shared memory):
//    a thread-block cluster of 8 CTAs per unit, each owning a contiguous slice
//    of the rows.  Per iteration the CTAs exchange per-head (max, sum) and
//    their local argmin through distributed shared memory (two cluster
//    barriers).  Each row keeps y_j = C k_j; a Welford fold changes C by
//    C' = a C + b u dk^T (a = n/(n+1), b = 1/(n+1), u = v* - mu_v', dk =
//    k* - mu_k), so y_j' = a y_j + b u (dk . k_j) costs O(d) per row instead
//    of O(d^2).  The clamp stays exact: every iteration lists the entries with
//    0 < |n C_ab| < tau and subtracts C_ab k_jb from y_ja for them; if there
//    are more than kMaxClamp such entries that iteration computes C' k_j
//    directly.
//  - evict_kernel (fallback for larger capacities): one CTA per unit,
//    recomputing C' k_j for every row every iteration.
#include <cooperative_groups.h>

#include "common.cuh"
#include "kernels.h"

namespace cg = cooperative_groups;

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

constexpr int kCL = 8;          // CTAs per unit (one cluster)

// Bytes of staging per unit (K and V rows, positions), padded so that every
// unit's block starts on a 256-byte boundary.
__host__ __device__ inline size_t stage_stride(int cap, int D) {
  return align_up((size_t)cap * (4 * (size_t)D + 4), 256);
}
constexpr int kMaxClamp = 64;   // clamped entries corrected incrementally
constexpr size_t kSmemBudget = 220 * 1024;

template <int D, int G>
struct ClusterLayout {
  size_t Ct, Y, lg, kbuf, Ks, Vs, alive, total;
  __host__ __device__ ClusterLayout(int R, int kv) {
    size_t off = 0;
    Ct = off; off += (size_t)D * D * 4;
    Y = off; off += (size_t)R * D * 4;
    lg = off; off += align_up((size_t)G * R * 4, 16);
    kbuf = off; off += (size_t)kWarps * kRowsPerGroup * D * 4;
    Ks = off; off += kv ? (size_t)R * D * 2 : 0;
    Vs = off; off += kv ? (size_t)R * D * 2 : 0;
    alive = off; off += align_up((size_t)R, 16);
    total = off;
  }
};

template <int D, int G>
__global__ void __cluster_dims__(kCL, 1, 1) __launch_bounds__(kThreads)
    evict_cluster_kernel(const EvictArgs a) {
  constexpr int DPL = D / 32;
  extern __shared__ __align__(16) uint8_t dsmem[];
  const int R = a.rows_max;
  const ClusterLayout<D, G> lay(R, a.kv_smem);
  float* Ct = reinterpret_cast<float*>(dsmem + lay.Ct);      // Ct[c*D + r] = C[r][c]
  float* Y = reinterpret_cast<float*>(dsmem + lay.Y);        // [R][D] y_j = C k_j
  float* lg = reinterpret_cast<float*>(dsmem + lay.lg);      // [G][R] logits
  float* kbuf = reinterpret_cast<float*>(dsmem + lay.kbuf);  // [warps][4][D]
  uint8_t* alive = dsmem + lay.alive;                        // [R]
  __shared__ float s_mu_k[D], s_mu_v[D], s_dk[D], s_dv[D];
  __shared__ float s_q[G][D];
  __shared__ float s_red[kWarps][G];
  __shared__ float s_M[G], s_Z[G];
  __shared__ float ex_ml[2 * G];       // this CTA's per-head (max, sum), read by the cluster
  __shared__ unsigned long long ex_best;
  __shared__ int ex_cnt;
  __shared__ unsigned long long s_bestw[kWarps];
  __shared__ uint32_t s_zidx[kMaxClamp];
  __shared__ float s_zval[kMaxClamp];
  __shared__ int s_nz;

  cg::cluster_group cluster = cg::this_cluster();
  const int rank = static_cast<int>(cluster.block_rank());
  const int u = blockIdx.x / kCL;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const size_t row0 = (size_t)u * a.cap;
  __nv_bfloat16* Kg = reinterpret_cast<__nv_bfloat16*>(a.K) + row0 * D;
  __nv_bfloat16* Vg = reinterpret_cast<__nv_bfloat16*>(a.V) + row0 * D;
  int32_t* Pg = a.pos + row0;
  const int len_in = a.len[u];
  const int seen_in = a.seen[u];
  const bool has_new = a.k_new != nullptr;
  if (len_in < 0 || len_in > a.cap || (has_new && len_in + 1 > a.cap)) {
    if (rank == 0 && tid == 0) record_error(a.ws, MKV_ERR_CAPACITY, u);
    return;  // uniform over the cluster
  }
  const int len = len_in + (has_new ? 1 : 0);
  const int rows_per = (len + kCL - 1) / kCL;
  const int j0 = min(len, rank * rows_per), j1 = min(len, j0 + rows_per);
  const int nr = j1 - j0;
  if (has_new && len_in >= j0 && len_in < j1) {  // the owning CTA appends the token
    const __nv_bfloat16* kn = reinterpret_cast<const __nv_bfloat16*>(a.k_new) + (size_t)u * D;
    const __nv_bfloat16* vn = reinterpret_cast<const __nv_bfloat16*>(a.v_new) + (size_t)u * D;
    for (int i = tid; i < D; i += kThreads) {
      Kg[(size_t)len_in * D + i] = kn[i];
      Vg[(size_t)len_in * D + i] = vn[i];
    }
    if (tid == 0) Pg[len_in] = seen_in;
    __threadfence();
  }
  __syncthreads();  // the appended row is read back below by other threads
  if (len <= a.budget) {
    if (rank == 0 && tid == 0) {
      a.len[u] = len;
      a.seen[u] = seen_in + (has_new ? 1 : 0);
    }
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
  // this slice's rows (global or cached in shared memory)
  const __nv_bfloat16* Kr = Kg + (size_t)j0 * D;
  const __nv_bfloat16* Vr = Vg + (size_t)j0 * D;
  if (a.kv_smem) {
    __nv_bfloat16* Ks = reinterpret_cast<__nv_bfloat16*>(dsmem + lay.Ks);
    __nv_bfloat16* Vs = reinterpret_cast<__nv_bfloat16*>(dsmem + lay.Vs);
    for (int idx = tid; idx < nr * (D / 8); idx += kThreads) {
      reinterpret_cast<uint4*>(Ks)[idx] = reinterpret_cast<const uint4*>(Kr)[idx];
      reinterpret_cast<uint4*>(Vs)[idx] = reinterpret_cast<const uint4*>(Vr)[idx];
    }
    Kr = Ks;
    Vr = Vs;
  }
  for (int r = tid; r < R; r += kThreads) alive[r] = r < nr ? 1 : 0;
  if (tid == 0) s_nz = 0;
  __syncthreads();

  // logits and y_j = C k_j for the slice
  for (int r = warp; r < nr; r += kWarps) {
    float kf[DPL];
    load_bf16<DPL>(Kr + (size_t)r * D + lane * DPL, kf);
#pragma unroll
    for (int h = 0; h < G; ++h) {
      float acc = 0.f;
#pragma unroll
      for (int i = 0; i < DPL; ++i) acc = fmaf(s_q[h][lane * DPL + i], kf[i], acc);
      acc = warp_sum(acc);
      if (lane == 0) lg[h * R + r] = acc;
    }
  }
  float* kb = kbuf + warp * kRowsPerGroup * D;
  for (int g0 = warp * kRowsPerGroup; g0 < nr; g0 += kWarps * kRowsPerGroup) {
#pragma unroll
    for (int r = 0; r < kRowsPerGroup; ++r) {
      float kf[DPL];
      if (g0 + r < nr) {
        load_bf16<DPL>(Kr + (size_t)(g0 + r) * D + lane * DPL, kf);
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
#pragma unroll
        for (int i = 0; i < DPL; ++i) cv[i] = Ct[c * D + lane * DPL + i];
#pragma unroll
        for (int r = 0; r < kRowsPerGroup; ++r) {
          const float kc = kb[r * D + c];
#pragma unroll
          for (int i = 0; i < DPL; ++i) y[r][i] = fmaf(cv[i], kc, y[r][i]);
        }
      }
    }
#pragma unroll
    for (int r = 0; r < kRowsPerGroup; ++r)
      if (g0 + r < nr) {
#pragma unroll
        for (int i = 0; i < DPL; ++i) Y[(size_t)(g0 + r) * D + lane * DPL + i] = y[r][i];
      }
    __syncwarp();
  }
  // clamp list for the initial moments: entries with 0 < |n C_ab| < tau
  const float tau = a.tau;
  if (n > 0 && tau > 0.f) {
    const float nf = static_cast<float>(n);
    for (int idx = tid; idx < D * D; idx += kThreads) {
      const float c = Ct[idx];
      if (c != 0.f && fabsf(c * nf) < tau) {
        const int k = atomicAdd(&s_nz, 1);
        if (k < kMaxClamp) {
          s_zidx[k] = static_cast<uint32_t>(idx);
          s_zval[k] = c;
        }
      }
    }
  }
  __syncthreads();

  const int n_evict = len - a.budget;
  for (int e = 0; e < n_evict; ++e) {
    // ---- phase A: per-head softmax normaliser over the whole unit
    {
      float mx[G], zs[G];
#pragma unroll
      for (int h = 0; h < G; ++h) mx[h] = -INFINITY;
      for (int r = tid; r < nr; r += kThreads)
        if (alive[r]) {
#pragma unroll
          for (int h = 0; h < G; ++h) mx[h] = fmaxf(mx[h], lg[h * R + r]);
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
        s_M[tid] = m;
      }
      __syncthreads();
#pragma unroll
      for (int h = 0; h < G; ++h) zs[h] = 0.f;
      for (int r = tid; r < nr; r += kThreads)
        if (alive[r]) {
#pragma unroll
          for (int h = 0; h < G; ++h) zs[h] += expf(lg[h * R + r] - s_M[h]);
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
        ex_ml[tid] = s_M[tid];
        ex_ml[G + tid] = z;
      }
    }
    cluster.sync();
    if (tid < G) {
      float M = -INFINITY;
      for (int r = 0; r < kCL; ++r) M = fmaxf(M, cluster.map_shared_rank(ex_ml, r)[tid]);
      float Z = 0.f;
      for (int r = 0; r < kCL; ++r) {
        const float* rm = cluster.map_shared_rank(ex_ml, r);
        if (rm[tid] != -INFINITY) Z += rm[G + tid] * expf(rm[tid] - M);
      }
      s_M[tid] = M;
      s_Z[tid] = Z;
    }
    __syncthreads();

    // ---- phase B: scores of this slice, local argmin
    const float rs = (n > 0) ? scale : 0.f;
    const int nz = s_nz;
    const bool direct = nz > kMaxClamp;
    const float nf = static_cast<float>(n);
    unsigned long long best = ~0ull;
    for (int r = warp; r < nr; r += kWarps) {
      if (!alive[r]) continue;  // warp-uniform
      float yv[DPL], vf[DPL];
      load_bf16<DPL>(Vr + (size_t)r * D + lane * DPL, vf);
      if (!direct) {
#pragma unroll
        for (int i = 0; i < DPL; ++i) yv[i] = Y[(size_t)r * D + lane * DPL + i];
        for (int z = 0; z < nz; ++z) {  // y'_a -= C_ab k_b for clamped (a, b)
          const uint32_t idx = s_zidx[z];
          const int cb = static_cast<int>(idx / D), ra = static_cast<int>(idx % D);
          if (ra / DPL == lane) yv[ra % DPL] -= s_zval[z] * __bfloat162float(Kr[(size_t)r * D + cb]);
        }
      } else {
        float kf[DPL];
        load_bf16<DPL>(Kr + (size_t)r * D + lane * DPL, kf);
#pragma unroll
        for (int i = 0; i < DPL; ++i) yv[i] = 0.f;
        for (int c = 0; c < D; ++c) {
          const float kc = __shfl_sync(kFull, kf[c % DPL], c / DPL);
#pragma unroll
          for (int i = 0; i < DPL; ++i) {
            float cv = Ct[c * D + lane * DPL + i];
            cv = (fabsf(cv * nf) < tau) ? 0.f : cv;
            yv[i] = fmaf(cv, kc, yv[i]);
          }
        }
      }
      float ss = 0.f;
#pragma unroll
      for (int i = 0; i < DPL; ++i) {
        const float rr = vf[i] - s_mu_v[lane * DPL + i] - rs * yv[i];
        ss = fmaf(rr, rr, ss);
      }
      ss = warp_sum(ss);
      float alpha = 0.f;
#pragma unroll
      for (int h = 0; h < G; ++h) alpha += expf(lg[h * R + r] - s_M[h]) / s_Z[h];
      const float score = alpha * sqrtf(ss);
      const unsigned long long key =
          (static_cast<unsigned long long>(__float_as_uint(score)) << 32) | static_cast<unsigned>(j0 + r);
      best = key < best ? key : best;
    }
    best = shfl_min_u64(best);
    if (lane == 0) s_bestw[warp] = best;
    __syncthreads();
    if (tid == 0) {
      unsigned long long b = s_bestw[0];
      for (int w = 1; w < kWarps; ++w) b = s_bestw[w] < b ? s_bestw[w] : b;
      ex_best = b;
      s_nz = 0;
    }
    cluster.sync();
    unsigned long long gb = ~0ull;
    for (int r = 0; r < kCL; ++r) {
      const unsigned long long v = *cluster.map_shared_rank(&ex_best, r);
      gb = v < gb ? v : gb;
    }
    const int js = static_cast<int>(gb & 0xffffffffu);

    // ---- phase C: fold row j* into the moments, update y for the slice
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
    if (tid == 0 && js >= j0 && js < j1) alive[js - j0] = 0;
    __syncthreads();
    const float keep = static_cast<float>(n) / n1;
    const float inv = 1.f / n1;
    for (int idx = tid; idx < D * D; idx += kThreads) {
      const int c = idx / D, r = idx % D;  // Ct[c][r] = C[r][c]
      const float v = keep * Ct[idx] + inv * s_dv[r] * s_dk[c];
      Ct[idx] = v;
      if (tau > 0.f && v != 0.f && fabsf(v * n1) < tau) {
        const int k = atomicAdd(&s_nz, 1);
        if (k < kMaxClamp) {
          s_zidx[k] = static_cast<uint32_t>(idx);
          s_zval[k] = v;
        }
      }
    }
    for (int r = warp; r < nr; r += kWarps) {
      if (!alive[r]) continue;
      float kf[DPL];
      load_bf16<DPL>(Kr + (size_t)r * D + lane * DPL, kf);
      float dot = 0.f;
#pragma unroll
      for (int i = 0; i < DPL; ++i) dot = fmaf(s_dk[lane * DPL + i], kf[i], dot);
      dot = warp_sum(dot) * inv;
#pragma unroll
      for (int i = 0; i < DPL; ++i) {
        float* yp = Y + (size_t)r * D + lane * DPL + i;
        *yp = keep * *yp + dot * s_dv[lane * DPL + i];
      }
    }
    n += 1;
    __syncthreads();
  }

  // ---- ordered compaction across the cluster through the staging buffer
  {
    int cnt = 0;
    for (int r = tid; r < nr; r += kThreads) cnt += alive[r];
    cnt = static_cast<int>(warp_sum(static_cast<float>(cnt)));
    if (lane == 0) s_red[warp][0] = static_cast<float>(cnt);
    __syncthreads();
    if (tid == 0) {
      int c = 0;
      for (int w = 0; w < kWarps; ++w) c += static_cast<int>(s_red[w][0]);
      ex_cnt = c;
    }
  }
  cluster.sync();
  int base = 0;
  for (int r = 0; r < rank; ++r) base += *cluster.map_shared_rank(&ex_cnt, r);
  const int mine = ex_cnt;
  uint8_t* st = static_cast<uint8_t*>(a.stage) + (size_t)u * stage_stride(a.cap, D);
  __nv_bfloat16* SK = reinterpret_cast<__nv_bfloat16*>(st);
  __nv_bfloat16* SV = SK + (size_t)a.cap * D;
  int32_t* SP = reinterpret_cast<int32_t*>(SV + (size_t)a.cap * D);
  if (warp == 0) {
    int run = base;
    for (int c0 = 0; c0 < nr; c0 += 32) {
      const bool al = (c0 + lane < nr) && alive[c0 + lane];
      const unsigned m = __ballot_sync(kFull, al);
      if (al) SP[run + __popc(m & ((1u << lane) - 1u))] = Pg[j0 + c0 + lane];
      run += __popc(m);
    }
  }
  {
    // rows: each warp copies survivors; destination = base + rank among survivors
    for (int c0 = 0; c0 < nr; c0 += 32) {
      const bool al = (c0 + lane < nr) && alive[c0 + lane];
      const unsigned m = __ballot_sync(kFull, al);
      int before = 0;  // survivors in earlier chunks
      for (int c1 = 0; c1 < c0; c1 += 32) {
        const bool a1 = (c1 + lane < nr) && alive[c1 + lane];
        before += __popc(__ballot_sync(kFull, a1));
      }
      for (int bit = warp; bit < 32; bit += kWarps) {
        if (!((m >> bit) & 1u)) continue;
        const int r = c0 + bit;
        const int dst = base + before + __popc(m & ((1u << bit) - 1u));
        for (int i = lane; i < D / 8; i += 32) {
          reinterpret_cast<uint4*>(SK + (size_t)dst * D)[i] = reinterpret_cast<const uint4*>(Kr + (size_t)r * D)[i];
          reinterpret_cast<uint4*>(SV + (size_t)dst * D)[i] = reinterpret_cast<const uint4*>(Vr + (size_t)r * D)[i];
        }
      }
    }
  }
  __threadfence();
  cluster.sync();
  for (int idx = tid; idx < mine * (D / 8); idx += kThreads) {
    const int row = base + idx / (D / 8), i = idx % (D / 8);
    reinterpret_cast<uint4*>(Kg + (size_t)row * D)[i] = reinterpret_cast<const uint4*>(SK + (size_t)row * D)[i];
    reinterpret_cast<uint4*>(Vg + (size_t)row * D)[i] = reinterpret_cast<const uint4*>(SV + (size_t)row * D)[i];
  }
  for (int r = tid; r < mine; r += kThreads) Pg[base + r] = SP[base + r];
  if (rank == 0) {
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
      a.seen[u] = seen_in + (has_new ? 1 : 0);
    }
  }
}

template <int D, int G>
size_t cluster_smem(int cap, int* kv) {
  const int R = (cap + kCL - 1) / kCL;
  const size_t with_kv = ClusterLayout<D, G>(R, 1).total;
  if (with_kv <= kSmemBudget) {
    *kv = 1;
    return with_kv;
  }
  *kv = 0;
  return ClusterLayout<D, G>(R, 0).total;
}

template <int D, int G>
cudaError_t launch_dg(const EvictArgs& a0, cudaStream_t stream) {
  EvictArgs a = a0;
  int kv = 0;
  const size_t csm = cluster_smem<D, G>(a.cap, &kv);
  if (csm <= kSmemBudget) {
    a.rows_max = (a.cap + kCL - 1) / kCL;
    a.kv_smem = kv;
    cudaError_t e = cudaFuncSetAttribute(evict_cluster_kernel<D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(csm));
    if (e != cudaSuccess) return e;
    evict_cluster_kernel<D, G><<<a.batch * a.n_kv * kCL, kThreads, csm, stream>>>(a);
    return cudaGetLastError();
  }
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
  return kHeaderBytes + align_up(units * g.group * (size_t)capacity * sizeof(float), 256) +
         units * stage_stride(capacity, g.head_dim);
}

void evict_carve(EvictArgs& a, const mkv_geom& g, int32_t capacity, void* ws) {
  const size_t units = (size_t)g.batch * g.n_kv_heads;
  uint8_t* p = static_cast<uint8_t*>(ws);
  a.ws = ws;
  a.scratch = reinterpret_cast<float*>(p + kHeaderBytes);
  a.stage = p + kHeaderBytes + align_up(units * g.group * (size_t)capacity * sizeof(float), 256);
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
