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
// Three kernels compute the same thing, chosen by the capacity:
//  - evict_reg_kernel (row slices of up to 144 rows; described before it):
//    the state of the loop in registers, one block and one cluster barrier
//    per eviction;
//  - evict_cluster_kernel (larger slices that fit shared memory):
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
    if (a.y_len != nullptr) a.y_len[u] = 0;  // rows moved and the moments changed: no y row is current
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

constexpr int kCL = 8;           // CTAs per unit (one cluster)
constexpr int kCT = 1024;        // threads per CTA of the cluster kernel
constexpr int kCW = kCT / 32;    // warps per CTA
constexpr int kLPR = 8;          // lanes per row
constexpr int kRPW = 32 / kLPR;  // rows per warp per pass
constexpr int kRowsPerPass = kCW * kRPW;
constexpr int kMaxClamp = 64;    // clamped entries corrected incrementally
constexpr int kTW = 4;           // warps that run the 32x32 tile transposes
constexpr int kTWR = 8;          // the same in the register kernel
// dynamic shared memory available next to the kernel's ~30 KB of static arrays
constexpr size_t kSmemBudget = 192 * 1024;

// Bytes of staging per unit (K and V rows, positions), padded so that every
// unit's block starts on a 256-byte boundary.
__host__ __device__ inline size_t stage_stride(int cap, int D) {
  return align_up((size_t)cap * (4 * (size_t)D + 4), 256);
}

template <int D, int G>
struct ClusterLayout {
  size_t Ct, Y, lg, Ks, Vs, alive, total;
  // R rows per slice; cap rows per unit (logits and alive flags cover the unit)
  __host__ __device__ ClusterLayout(int R, int cap, int kv) {
    size_t off = 0;
    Ct = off; off += (size_t)D * D * 4;
    Y = off; off += (size_t)R * D * 4;
    lg = off; off += align_up((size_t)G * cap * 4, 16);
    Ks = off; off += kv ? (size_t)R * D * 2 : 0;
    Vs = off; off += kv ? (size_t)R * D * 2 : 0;
    alive = off; off += align_up((size_t)cap, 16);
    total = off;
  }
};

// A row is handled by a group of 8 lanes; lane q of the group owns the
// value/key dims of float4 chunks q, q+8, q+16, ... (NC = D/32 chunks), so
// the 8 lanes of a row touch 8 different bank groups.
template <int D>
__device__ __forceinline__ int chunk_dim(int q, int c) { return (q + 8 * c) * 4; }

__device__ __forceinline__ float group_sum(float v) {
  v += __shfl_xor_sync(kFull, v, 1);
  v += __shfl_xor_sync(kFull, v, 2);
  v += __shfl_xor_sync(kFull, v, 4);
  return v;
}

template <int D>
__device__ __forceinline__ void load4_bf16(const __nv_bfloat16* p, float* o) { load_bf16<4>(p, o); }

// Vectors of N floats in shared memory (aligned to 4N bytes).
template <int N>
__device__ __forceinline__ void ld_vec(const float* p, float* v) {
  if constexpr (N == 4) {
    const float4 t = *reinterpret_cast<const float4*>(p);
    v[0] = t.x; v[1] = t.y; v[2] = t.z; v[3] = t.w;
  } else {
    const float2 t = *reinterpret_cast<const float2*>(p);
    v[0] = t.x; v[1] = t.y;
  }
}
template <int N>
__device__ __forceinline__ void st_vec(float* p, const float* v) {
  if constexpr (N == 4) *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  else *reinterpret_cast<float2*>(p) = make_float2(v[0], v[1]);
}

template <int D, int G>
__global__ void __cluster_dims__(kCL, 1, 1) __launch_bounds__(kCT, 1)
    evict_cluster_kernel(const EvictArgs a) {
  constexpr int NC = D / 32;
  constexpr int DPL = D / 32;  // consecutive C columns per thread in the rank-1 update of Ct
  extern __shared__ __align__(16) uint8_t dsmem[];
  const int R = a.rows_max;
  const ClusterLayout<D, G> lay(R, a.cap, a.kv_smem);
  float* Ct = reinterpret_cast<float*>(dsmem + lay.Ct);  // Ct[c*D + r] = C[r][c]
  float* Y = reinterpret_cast<float*>(dsmem + lay.Y);    // [R][D] y_j = C k_j of this slice
  float* lg = reinterpret_cast<float*>(dsmem + lay.lg);  // [G][cap] logits of every row of the unit
  uint8_t* alive_all = dsmem + lay.alive;                // [cap] alive flags of the unit
  __shared__ __align__(16) float s_mu_k[D];
  __shared__ __align__(16) float s_mu_v[D];
  __shared__ __align__(16) float s_q[G][D];
  __shared__ __align__(16) float s_dk[D];
  __shared__ __align__(16) float s_dv[D];
  __shared__ float s_red[kCW][G];
  __shared__ double s_zpart[kCW][G];
  __shared__ float s_M[G], s_invZ[G];
  __shared__ float s_keep;
  __shared__ int s_js;
  // this CTA's best (score, row) key, reduced by atomicMin; and the mailbox
  // that every rank writes its key and candidate row into (double-buffered by
  // iteration parity)
  __shared__ unsigned long long s_best[2];
  __shared__ unsigned long long mail_key[2][kCL];
  __shared__ __align__(16) __nv_bfloat16 mail_row[2][kCL][2 * D];
  __shared__ int ex_cnt;
  __shared__ uint32_t s_zidx[2][kMaxClamp];
  __shared__ float s_zval[2][kMaxClamp];
  __shared__ int s_nz[2];
  __shared__ float s_tile[kTW][32 * 33];  // transpose staging (setup / write-back)

  cg::cluster_group cluster = cg::this_cluster();
  const int rank = static_cast<int>(cluster.block_rank());
  const int u = blockIdx.x / kCL;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int q = lane & 7;                      // lane within its row group
  const int rsub = warp * kRPW + (lane >> 3);  // row of this group within a pass
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
    for (int i = tid; i < D; i += kCT) {
      Kg[(size_t)len_in * D + i] = kn[i];
      Vg[(size_t)len_in * D + i] = vn[i];
    }
    if (tid == 0) Pg[len_in] = seen_in;
    __threadfence();
  }
  __syncthreads();
  if (len <= a.budget) {
    if (rank == 0 && tid == 0) {
      a.len[u] = len;
      a.seen[u] = seen_in + (has_new ? 1 : 0);
    }
    return;
  }
  // other CTAs' rows (the appended one included) are read below
  cluster.sync();

  int n = a.n[u];
  {
    // Ct[c][r] = C[r][c]: each warp moves 32x32 tiles through a padded buffer
    // so that both the global reads and the shared-memory writes are dense
    float* tb = s_tile[warp % kTW];
    for (int t = warp; warp < kTW && t < (D / 32) * (D / 32); t += kTW) {
      const int r0 = (t / (D / 32)) * 32, c0 = (t % (D / 32)) * 32;
      for (int i = 0; i < 32; ++i)
        tb[i * 33 + lane] = (n > 0) ? a.C[(size_t)u * D * D + (size_t)(r0 + i) * D + c0 + lane] : 0.f;
      __syncwarp();
      for (int i = 0; i < 32; ++i) Ct[(size_t)(c0 + i) * D + r0 + lane] = tb[lane * 33 + i];
      __syncwarp();
    }
  }
  for (int i = tid; i < D; i += kCT) {
    s_mu_k[i] = (n > 0) ? a.mu_k[(size_t)u * D + i] : 0.f;
    s_mu_v[i] = (n > 0) ? a.mu_v[(size_t)u * D + i] : 0.f;
  }
  const float scale = rsqrtf(static_cast<float>(D));
  const __nv_bfloat16* qg = reinterpret_cast<const __nv_bfloat16*>(a.q) + (size_t)u * G * D;
  for (int i = tid; i < G * D; i += kCT) s_q[i / D][i % D] = __bfloat162float(qg[i]) * scale;
  const __nv_bfloat16* Kr = Kg + (size_t)j0 * D;
  const __nv_bfloat16* Vr = Vg + (size_t)j0 * D;
  if (a.kv_smem) {
    __nv_bfloat16* Ks = reinterpret_cast<__nv_bfloat16*>(dsmem + lay.Ks);
    __nv_bfloat16* Vs = reinterpret_cast<__nv_bfloat16*>(dsmem + lay.Vs);
    for (int idx = tid; idx < nr * (D / 8); idx += kCT) {
      reinterpret_cast<uint4*>(Ks)[idx] = reinterpret_cast<const uint4*>(Kr)[idx];
      reinterpret_cast<uint4*>(Vs)[idx] = reinterpret_cast<const uint4*>(Vr)[idx];
    }
    Kr = Ks;
    Vr = Vs;
  }
  for (int j = tid; j < a.cap; j += kCT) alive_all[j] = j < len ? 1 : 0;
  if (tid == 0) {
    s_nz[0] = s_nz[1] = 0;
    s_best[0] = s_best[1] = ~0ull;
  }
  __syncthreads();
  const uint8_t* alive = alive_all + j0;  // this slice's flags

  // ---- logits of every row of the unit (8 lanes per row, read from global)
  for (int base = 0; base < len; base += kRowsPerPass) {
    const int j = base + rsub;
    const bool ok = j < len;
    float kf[NC][4];
#pragma unroll
    for (int c = 0; c < NC; ++c) {
      if (ok) load4_bf16<D>(Kg + (size_t)j * D + chunk_dim<D>(q, c), kf[c]);
      else kf[c][0] = kf[c][1] = kf[c][2] = kf[c][3] = 0.f;
    }
#pragma unroll
    for (int h = 0; h < G; ++h) {
      float acc = 0.f;
#pragma unroll
      for (int c = 0; c < NC; ++c) {
        const float4 q4 = *reinterpret_cast<const float4*>(&s_q[h][chunk_dim<D>(q, c)]);
        acc = fmaf(q4.x, kf[c][0], fmaf(q4.y, kf[c][1], fmaf(q4.z, kf[c][2], fmaf(q4.w, kf[c][3], acc))));
      }
      acc = group_sum(acc);
      if (ok && q == 0) lg[h * a.cap + j] = acc;
    }
  }
  __syncthreads();
  // softmax is shift-invariant: keep e_hj = exp(l_hj - M0_h) with M0_h the
  // largest logit of the unit at the start, so that every iteration's
  // normaliser is a plain sum over the surviving rows
  {
    float mx[G];
#pragma unroll
    for (int h = 0; h < G; ++h) mx[h] = -INFINITY;
    for (int jj = tid; jj < len; jj += kCT)
#pragma unroll
      for (int h = 0; h < G; ++h) mx[h] = fmaxf(mx[h], lg[h * a.cap + jj]);
#pragma unroll
    for (int h = 0; h < G; ++h) {
      mx[h] = warp_max(mx[h]);
      if (lane == 0) s_red[warp][h] = mx[h];
    }
    __syncthreads();
    if (warp == 0) {
#pragma unroll
      for (int h = 0; h < G; ++h) {
        const float m = warp_max(s_red[lane][h]);
        if (lane == 0) s_M[h] = m;
      }
    }
    __syncthreads();
    for (int jj = tid; jj < len; jj += kCT)
#pragma unroll
      for (int h = 0; h < G; ++h) lg[h * a.cap + jj] = expf(lg[h * a.cap + jj] - s_M[h]);
  }
  // ---- y_j = C k_j for this slice
  for (int base = 0; base < nr; base += kRowsPerPass) {
    const int r = base + rsub;
    const bool ok = r < nr;
    if (n > 0) {
      float y[NC][4];
#pragma unroll
      for (int c = 0; c < NC; ++c) y[c][0] = y[c][1] = y[c][2] = y[c][3] = 0.f;
      if (ok) {
        for (int kc = 0; kc < D; ++kc) {
          const float kv = __bfloat162float(Kr[(size_t)r * D + kc]);
#pragma unroll
          for (int c = 0; c < NC; ++c) {
            const float4 c4 = *reinterpret_cast<const float4*>(Ct + kc * D + chunk_dim<D>(q, c));
            y[c][0] = fmaf(c4.x, kv, y[c][0]);
            y[c][1] = fmaf(c4.y, kv, y[c][1]);
            y[c][2] = fmaf(c4.z, kv, y[c][2]);
            y[c][3] = fmaf(c4.w, kv, y[c][3]);
          }
        }
      }
      if (ok) {
#pragma unroll
        for (int c = 0; c < NC; ++c)
          *reinterpret_cast<float4*>(Y + (size_t)r * D + chunk_dim<D>(q, c)) = make_float4(y[c][0], y[c][1], y[c][2], y[c][3]);
      }
    } else if (ok) {
#pragma unroll
      for (int c = 0; c < NC; ++c)
        *reinterpret_cast<float4*>(Y + (size_t)r * D + chunk_dim<D>(q, c)) = make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
  // clamp list for the initial moments: entries with 0 < |n C_ab| < tau
  // (iteration e reads list e & 1; the fold before it builds that list)
  const float tau = a.tau;
  if (n > 0 && tau > 0.f) {
    const float nf = static_cast<float>(n);
    for (int idx = tid; idx < D * D; idx += kCT) {
      const float c = Ct[idx];
      if (c != 0.f && fabsf(c * nf) < tau) {
        const int k = atomicAdd(&s_nz[0], 1);
        if (k < kMaxClamp) {
          s_zidx[0][k] = static_cast<uint32_t>(idx);
          s_zval[0][k] = c;
        }
      }
    }
  }
  // per-head normaliser Z_h = sum of e_hj over the surviving rows, kept in
  // double by warp 0 (lane h) and decremented as rows are evicted
  double zd = 0.0;
  {
    double zs[G];
#pragma unroll
    for (int h = 0; h < G; ++h) zs[h] = 0.0;
    for (int jj = tid; jj < len; jj += kCT)
#pragma unroll
      for (int h = 0; h < G; ++h) zs[h] += static_cast<double>(lg[h * a.cap + jj]);
#pragma unroll
    for (int h = 0; h < G; ++h) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) zs[h] += __shfl_xor_sync(kFull, zs[h], o);
      if (lane == 0) s_zpart[warp][h] = zs[h];
    }
    __syncthreads();
    if (warp == 0 && lane < G) {
      for (int w = 0; w < kCW; ++w) zd += s_zpart[w][lane];
      s_invZ[lane] = 1.f / static_cast<float>(zd);
    }
  }
  __syncthreads();

  const int n_evict = len - a.budget;
  for (int e = 0;; ++e) {
    const int par = e & 1;
    // ---- fold the previous eviction into C (building clamp list par) and
    // into y_j of this slice: C' = keep C + dk dv^T, y_j' = keep y_j + (dk . k_j) dv
    if (e > 0) {
      const float nf = static_cast<float>(n);
      const float keep = s_keep;
      const float thr = tau / nf;  // |C_ab| < tau / n  <=>  |n C_ab| < tau
#pragma unroll
      for (int k = 0; k < D * D / DPL / kCT; ++k) {
        const int iv = k * kCT + tid;  // Ct[c][lane*DPL ...] with c = iv / 32
        const int c = iv >> 5;
        const float kd = s_dk[c];
        float v[DPL], dv[DPL];
        ld_vec<DPL>(Ct + (size_t)iv * DPL, v);
        ld_vec<DPL>(s_dv + lane * DPL, dv);
        bool any = false;
#pragma unroll
        for (int i = 0; i < DPL; ++i) {
          v[i] = fmaf(keep, v[i], kd * dv[i]);
          any |= fabsf(v[i]) < thr;
        }
        st_vec<DPL>(Ct + (size_t)iv * DPL, v);
        if (any) {
#pragma unroll
          for (int i = 0; i < DPL; ++i)
            if (v[i] != 0.f && fabsf(v[i] * nf) < tau) {
              const int slot = atomicAdd(&s_nz[par], 1);
              if (slot < kMaxClamp) {
                s_zidx[par][slot] = static_cast<uint32_t>(iv * DPL + i);
                s_zval[par][slot] = v[i];
              }
            }
        }
      }
      for (int base = 0; base < nr; base += kRowsPerPass) {
        const int r = base + rsub;
        const bool ok = (r < nr) && alive[r];
        float dot = 0.f;
        if (ok) {
#pragma unroll
          for (int c = 0; c < NC; ++c) {
            const int d0 = chunk_dim<D>(q, c);
            float kf[4];
            load4_bf16<D>(Kr + (size_t)r * D + d0, kf);
            const float4 k4 = *reinterpret_cast<const float4*>(s_dk + d0);
            dot = fmaf(k4.x, kf[0], fmaf(k4.y, kf[1], fmaf(k4.z, kf[2], fmaf(k4.w, kf[3], dot))));
          }
        }
        dot = group_sum(dot);
        if (ok) {
#pragma unroll
          for (int c = 0; c < NC; ++c) {
            const int d0 = chunk_dim<D>(q, c);
            float4* yp = reinterpret_cast<float4*>(Y + (size_t)r * D + d0);
            float4 y4 = *yp;
            const float4 dv = *reinterpret_cast<const float4*>(s_dv + d0);
            y4.x = fmaf(keep, y4.x, dot * dv.x);
            y4.y = fmaf(keep, y4.y, dot * dv.y);
            y4.z = fmaf(keep, y4.z, dot * dv.z);
            y4.w = fmaf(keep, y4.w, dot * dv.w);
            *yp = y4;
          }
        }
      }
    }
    __syncthreads();
    if (e == n_evict) break;  // uniform over the cluster

    // ---- scores of this slice (8 lanes per row), block minimum of the keys
    {
      const float rs = (n > 0) ? scale : 0.f;
      const int nz = s_nz[par];
      const bool direct = nz > kMaxClamp;
      const float nf = static_cast<float>(n);
      unsigned long long best = ~0ull;
      for (int base = 0; base < nr; base += kRowsPerPass) {
        const int r = base + rsub;
        const bool ok = (r < nr) && alive[r];
        float ss = 0.f;
        if (ok) {
          if (!direct) {
#pragma unroll
            for (int c = 0; c < NC; ++c) {
              const int d0 = chunk_dim<D>(q, c);
              float4 y4 = *reinterpret_cast<const float4*>(Y + (size_t)r * D + d0);
              for (int z = 0; z < nz; ++z) {  // y'_a -= C_ab k_b for clamped (a, b)
                const int kb = static_cast<int>(s_zidx[par][z] / D), va = static_cast<int>(s_zidx[par][z] % D);
                if (va >= d0 && va < d0 + 4) {
                  const float corr = s_zval[par][z] * __bfloat162float(Kr[(size_t)r * D + kb]);
                  const int o = va - d0;
                  if (o == 0) y4.x -= corr;
                  else if (o == 1) y4.y -= corr;
                  else if (o == 2) y4.z -= corr;
                  else y4.w -= corr;
                }
              }
              float vf[4];
              load4_bf16<D>(Vr + (size_t)r * D + d0, vf);
              const float4 m4 = *reinterpret_cast<const float4*>(s_mu_v + d0);
              const float r0 = vf[0] - m4.x - rs * y4.x, r1 = vf[1] - m4.y - rs * y4.y;
              const float r2 = vf[2] - m4.z - rs * y4.z, r3 = vf[3] - m4.w - rs * y4.w;
              ss = fmaf(r0, r0, fmaf(r1, r1, fmaf(r2, r2, fmaf(r3, r3, ss))));
            }
          } else {
            float y[NC][4];
#pragma unroll
            for (int c = 0; c < NC; ++c) y[c][0] = y[c][1] = y[c][2] = y[c][3] = 0.f;
            for (int kc = 0; kc < D; ++kc) {
              const float kv = __bfloat162float(Kr[(size_t)r * D + kc]);
#pragma unroll
              for (int c = 0; c < NC; ++c) {
                const float4 c4 = *reinterpret_cast<const float4*>(Ct + kc * D + chunk_dim<D>(q, c));
                y[c][0] = fmaf((fabsf(c4.x * nf) < tau) ? 0.f : c4.x, kv, y[c][0]);
                y[c][1] = fmaf((fabsf(c4.y * nf) < tau) ? 0.f : c4.y, kv, y[c][1]);
                y[c][2] = fmaf((fabsf(c4.z * nf) < tau) ? 0.f : c4.z, kv, y[c][2]);
                y[c][3] = fmaf((fabsf(c4.w * nf) < tau) ? 0.f : c4.w, kv, y[c][3]);
              }
            }
#pragma unroll
            for (int c = 0; c < NC; ++c) {
              const int d0 = chunk_dim<D>(q, c);
              float vf[4];
              load4_bf16<D>(Vr + (size_t)r * D + d0, vf);
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                const float rr = vf[i] - s_mu_v[d0 + i] - rs * y[c][i];
                ss = fmaf(rr, rr, ss);
              }
            }
          }
        }
        ss = group_sum(ss);
        if (ok && q == 0) {
          float alpha = 0.f;
#pragma unroll
          for (int h = 0; h < G; ++h) alpha = fmaf(lg[h * a.cap + j0 + r], s_invZ[h], alpha);
          const float score = alpha * sqrtf(ss);
          const unsigned long long key =
              (static_cast<unsigned long long>(__float_as_uint(score)) << 32) | static_cast<unsigned>(j0 + r);
          best = key < best ? key : best;
        }
      }
      best = shfl_min_u64(best);
      if (lane == 0 && best != ~0ull) atomicMin(&s_best[par], best);
      if (tid == 0) s_nz[par ^ 1] = 0;  // list par^1 was last read one iteration ago
    }
    __syncthreads();

    // ---- warp 0 posts this CTA's key and candidate row into every rank's
    // mailbox slot [par][rank]; one cluster barrier publishes them all
    if (warp == 0) {
      const unsigned long long b = s_best[par];
      const int jb = (b == ~0ull) ? -1 : static_cast<int>(b & 0xffffffffu) - j0;
      if (lane < kCL) *cluster.map_shared_rank(&mail_key[par][rank], lane) = b;
      if (jb >= 0 && lane < D / 4) {  // lanes 0..D/8-1 carry k, the next D/8 carry v
        const bool is_v = lane >= D / 8;
        const int i = is_v ? lane - D / 8 : lane;
        const uint4 w = reinterpret_cast<const uint4*>((is_v ? Vr : Kr) + (size_t)jb * D)[i];
#pragma unroll
        for (int rk = 0; rk < kCL; ++rk)
          reinterpret_cast<uint4*>(cluster.map_shared_rank(&mail_row[par][rank][is_v ? D : 0], rk))[i] = w;
      }
      if (lane == 0) s_best[par] = ~0ull;  // next used two iterations on
    }
    cluster.sync();

    // ---- warp 0: the cluster's minimum key, Welford fold of that row (Eq. app_update)
    if (warp == 0) {
      unsigned long long b = (lane < kCL) ? mail_key[par][lane] : ~0ull;
      int w = lane;
#pragma unroll
      for (int o = 4; o > 0; o >>= 1) {
        const unsigned long long b2 = __shfl_xor_sync(kFull, b, o);
        const int w2 = __shfl_xor_sync(kFull, w, o);
        if (b2 < b || (b2 == b && w2 < w)) {
          b = b2;
          w = w2;
        }
      }
      b = __shfl_sync(kFull, b, 0);
      w = __shfl_sync(kFull, w, 0);
      const int js = (b == ~0ull) ? -1 : static_cast<int>(b & 0xffffffffu);
      if (js >= 0) {
        const float inv = 1.f / static_cast<float>(n + 1);
        for (int d = lane; d < D; d += 32) {
          const float kx = __bfloat162float(mail_row[par][w][d]);
          const float vx = __bfloat162float(mail_row[par][w][D + d]);
          const float dk = kx - s_mu_k[d];
          s_mu_k[d] = fmaf(dk, inv, s_mu_k[d]);
          const float mvn = fmaf(vx - s_mu_v[d], inv, s_mu_v[d]);
          s_mu_v[d] = mvn;
          s_dk[d] = dk * inv;  // scaled by 1/(n+1) for the rank-1 terms
          s_dv[d] = vx - mvn;
        }
        if (lane < G) {
          zd -= static_cast<double>(lg[lane * a.cap + js]);
          s_invZ[lane] = 1.f / static_cast<float>(zd);
        }
        if (lane == 0) {
          alive_all[js] = 0;
          s_keep = static_cast<float>(n) * inv;
        }
      }
      if (lane == 0) {
        if (js < 0) record_error(a.ws, MKV_ERR_INVALID_ARG, u);
        s_js = js;
      }
    }
    __syncthreads();
    if (s_js < 0) break;  // uniform: every rank read the same keys
    n += 1;
  }

  // ---- ordered compaction across the cluster through the staging buffer
  {
    int cnt = 0;
    for (int r = tid; r < nr; r += kCT) cnt += alive[r];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(kFull, cnt, o);
    if (lane == 0) s_red[warp][0] = static_cast<float>(cnt);
    __syncthreads();
    if (tid == 0) {
      int c = 0;
      for (int w = 0; w < kCW; ++w) c += static_cast<int>(s_red[w][0]);
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
  for (int c0 = 0; c0 < nr; c0 += 32) {
    // warp w moves row c0 + w of this chunk (32 warps = 32 rows)
    const bool al = (c0 + lane < nr) && alive[c0 + lane];
    const unsigned m = __ballot_sync(kFull, al);
    int before = 0;  // survivors in earlier chunks
    for (int c1 = 0; c1 < c0; c1 += 32) {
      const bool a1 = (c1 + lane < nr) && alive[c1 + lane];
      before += __popc(__ballot_sync(kFull, a1));
    }
    const int bit = warp;
    if ((m >> bit) & 1u) {
      const int r = c0 + bit;
      const int dst = base + before + __popc(m & ((1u << bit) - 1u));
      for (int i = lane; i < D / 8; i += 32) {
        reinterpret_cast<uint4*>(SK + (size_t)dst * D)[i] = reinterpret_cast<const uint4*>(Kr + (size_t)r * D)[i];
        reinterpret_cast<uint4*>(SV + (size_t)dst * D)[i] = reinterpret_cast<const uint4*>(Vr + (size_t)r * D)[i];
      }
      if (lane == 0) SP[dst] = Pg[j0 + r];
    }
  }
  __threadfence();
  cluster.sync();
  for (int idx = tid; idx < mine * (D / 8); idx += kCT) {
    const int row = base + idx / (D / 8), i = idx % (D / 8);
    reinterpret_cast<uint4*>(Kg + (size_t)row * D)[i] = reinterpret_cast<const uint4*>(SK + (size_t)row * D)[i];
    reinterpret_cast<uint4*>(Vg + (size_t)row * D)[i] = reinterpret_cast<const uint4*>(SV + (size_t)row * D)[i];
  }
  for (int r = tid; r < mine; r += kCT) Pg[base + r] = SP[base + r];
  if (rank == 0) {
    float* tb = s_tile[warp % kTW];
    for (int t = warp; warp < kTW && t < (D / 32) * (D / 32); t += kTW) {
      const int c0 = (t / (D / 32)) * 32, r0 = (t % (D / 32)) * 32;
      for (int i = 0; i < 32; ++i) tb[i * 33 + lane] = Ct[(size_t)(c0 + i) * D + r0 + lane];
      __syncwarp();
      for (int i = 0; i < 32; ++i) a.C[(size_t)u * D * D + (size_t)(r0 + i) * D + c0 + lane] = tb[lane * 33 + i];
      __syncwarp();
    }
    for (int i = tid; i < D; i += kCT) {
      a.mu_k[(size_t)u * D + i] = s_mu_k[i];
      a.mu_v[(size_t)u * D + i] = s_mu_v[i];
    }
    if (tid == 0) {
      a.n[u] = n;
      a.len[u] = a.budget;
      a.seen[u] = seen_in + (has_new ? 1 : 0);
      if (a.y_len != nullptr) a.y_len[u] = 0;  // rows moved and the moments changed: no y row is current
    }
  }
}

// ---------------------------------------------------------------------------
// Register-resident cluster kernel, used while a row slice has at most
// kRW * RPW rows.  8 CTAs of 512 threads per unit (one cluster); warp w of a
// CTA owns the slice rows w, w + 16, ... and lane l owns the dims
// [l*DPL, (l+1)*DPL) of each.  State in the raw co-moment form S_tilde = n C:
// y_j = S_tilde k_j of the warp's rows stays in registers, and so does a
// 1/512 share of S_tilde (rows a of the lane's dims, columns c = w + 16 i),
// which every iteration folds and scans for the clamp list.  Set-up: each CTA
// takes the logits and softmax (max, sum) of its own rows, and one cluster
// exchange gives the unit's maximum and normaliser.  Every thread computes the
// Welford fold of its own dims from the evicted row, so the only barriers of
// an iteration are one block barrier (the block's minimum key) and one
// cluster barrier (every CTA's key, candidate row and its softmax terms,
// written into every CTA's mailbox beforehand).  Scores are computed assuming
// an empty clamp list; when the list is not empty they are recomputed with it.
constexpr int kRT = 512;       // threads per CTA
constexpr int kRW = kRT / 32;  // warps per CTA

template <int D, int G>
struct RegLayout {
  size_t Ct, lg, Ks, Vs, alive, total;
  __host__ __device__ RegLayout(int R, int cap, int kv) {
    size_t off = 0;
    Ct = off; off += (size_t)D * D * 4;
    lg = off; off += align_up((size_t)G * R * 4, 16);
    Ks = off; off += kv ? (size_t)R * D * 2 : 0;
    Vs = off; off += kv ? (size_t)R * D * 2 : 0;
    alive = off; off += align_up((size_t)cap, 16);
    total = off;
  }
};

// Butterfly sums of N independent values across the warp (every lane gets them).
template <int N>
__device__ __forceinline__ void warp_sum_n(float (&v)[N]) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1)
#pragma unroll
    for (int i = 0; i < N; ++i) v[i] += __shfl_xor_sync(kFull, v[i], o);
}

// One round of a transposing butterfly: lanes with bit o set keep the upper
// W values, the others the lower W, and each adds its partner's copy.
template <int W>
__device__ __forceinline__ void tsum_round(float* v, int lane, int o) {
  const bool hi = (lane & o) != 0;
#pragma unroll
  for (int i = 0; i < W; ++i) {
    const float send = hi ? v[i] : v[i + W];
    const float keep = hi ? v[i + W] : v[i];
    v[i] = keep + __shfl_xor_sync(kFull, send, o);
  }
}

// Warp sums of P (8 or 16) values per lane in P - 1 + 5 - log2(P) shuffles:
// returns, in every lane, the sum over the warp of v[lane >> (5 - log2 P)].
template <int P>
__device__ __forceinline__ float transpose_sum(float (&v)[P], int lane) {
  static_assert(P == 8 || P == 16, "8 or 16 values");
  if constexpr (P == 16) tsum_round<8>(v, lane, 16);
  tsum_round<4>(v, lane, P == 16 ? 8 : 16);
  tsum_round<2>(v, lane, P == 16 ? 4 : 8);
  tsum_round<1>(v, lane, P == 16 ? 2 : 4);
  float r = v[0];
#pragma unroll
  for (int o = (P == 16 ? 1 : 2); o >= 1; o >>= 1) r += __shfl_xor_sync(kFull, r, o);
  return r;
}

template <int N>
__device__ __forceinline__ float select_n(const float (&v)[N], int i) {
  float r = v[0];
#pragma unroll
  for (int k = 1; k < N; ++k) r = (i == k) ? v[k] : r;
  return r;
}

template <int D, int G, int RPW>
__global__ void __cluster_dims__(kCL, 1, 1) __launch_bounds__(kRT, 1)
    evict_reg_kernel(const EvictArgs a) {
  constexpr int NC = D / 32;   // float4 chunks per row for 8-lane row groups (set-up)
  constexpr int DPL = D / 32;  // dims per lane
  constexpr int CJ = D / kRW;  // C columns per thread
  constexpr int kRP = kRW * (32 / kLPR);  // rows per pass of 8-lane groups
  extern __shared__ __align__(16) uint8_t dsmem[];
  const int R = a.rows_max;
  const RegLayout<D, G> lay(R, a.cap, a.kv_smem);
  float* Ct = reinterpret_cast<float*>(dsmem + lay.Ct);  // Ct[c*D + a] = C[a][c] (set-up, direct mode, write-back)
  float* lg = reinterpret_cast<float*>(dsmem + lay.lg);  // [G][R] e_hj of this CTA's rows
  uint8_t* alive_all = dsmem + lay.alive;
  __shared__ __align__(16) float s_mu_k[D];
  __shared__ __align__(16) float s_mu_v[D];
  __shared__ __align__(16) float s_q[G][D];
  __shared__ float s_red[kRW][G];
  __shared__ float s_zpart[kRW][G];
  __shared__ float s_M[G];        // this CTA's largest logit per head (read remotely), then the unit's
  __shared__ float s_Z[G];        // this CTA's sum of exp(l - s_M) per head (read remotely)
  __shared__ float mail_e[2][kCL][G];  // e_h of each CTA's candidate row
  __shared__ unsigned long long s_best[2];
  __shared__ unsigned long long mail_key[2][kCL];
  __shared__ __align__(16) __nv_bfloat16 mail_row[2][kCL][2 * D];
  __shared__ int ex_cnt;
  __shared__ uint32_t s_zidx[kMaxClamp];
  __shared__ float s_zval[kMaxClamp];
  __shared__ int s_nz;
  __shared__ float s_tile[kTWR][32 * 33];

  cg::cluster_group cluster = cg::this_cluster();
  const int rank = static_cast<int>(cluster.block_rank());
  const int u = blockIdx.x / kCL;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int q = lane & 7;
  const int rsub = warp * (32 / kLPR) + (lane >> 3);
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
  // rows 0..y_cur-1 of the cache's y rows are current (none without them)
  const int y_cur = (a.Y != nullptr && a.y_len != nullptr) ? max(0, min(a.y_len[u], len_in)) : 0;
  const int rows_per = (len + kCL - 1) / kCL;
  const int j0 = min(len, rank * rows_per), j1 = min(len, j0 + rows_per);
  const int nr = j1 - j0;
  if (has_new && len_in >= j0 && len_in < j1) {  // the owning CTA appends the token
    const __nv_bfloat16* kn = reinterpret_cast<const __nv_bfloat16*>(a.k_new) + (size_t)u * D;
    const __nv_bfloat16* vn = reinterpret_cast<const __nv_bfloat16*>(a.v_new) + (size_t)u * D;
    for (int i = tid; i < D; i += kRT) {
      Kg[(size_t)len_in * D + i] = kn[i];
      Vg[(size_t)len_in * D + i] = vn[i];
    }
    if (tid == 0) Pg[len_in] = seen_in;
    __threadfence();
  }
  __syncthreads();
  if (len <= a.budget) {
    if (rank == 0 && tid == 0) {
      a.len[u] = len;
      a.seen[u] = seen_in + (has_new ? 1 : 0);
    }
    return;
  }
  // other CTAs' rows (the appended one included) are read below
  cluster.sync();

  int n = a.n[u];
  {
    float* tb = s_tile[warp % kTWR];
    for (int t = warp; warp < kTWR && t < (D / 32) * (D / 32); t += kTWR) {
      const int r0 = (t / (D / 32)) * 32, c0 = (t % (D / 32)) * 32;
      for (int i = 0; i < 32; ++i)
        tb[i * 33 + lane] = (n > 0) ? a.C[(size_t)u * D * D + (size_t)(r0 + i) * D + c0 + lane] : 0.f;
      __syncwarp();
      for (int i = 0; i < 32; ++i) Ct[(size_t)(c0 + i) * D + r0 + lane] = tb[lane * 33 + i];
      __syncwarp();
    }
  }
  for (int i = tid; i < D; i += kRT) {
    s_mu_k[i] = (n > 0) ? a.mu_k[(size_t)u * D + i] : 0.f;
    s_mu_v[i] = (n > 0) ? a.mu_v[(size_t)u * D + i] : 0.f;
  }
  const float scale = rsqrtf(static_cast<float>(D));
  const __nv_bfloat16* qg = reinterpret_cast<const __nv_bfloat16*>(a.q) + (size_t)u * G * D;
  for (int i = tid; i < G * D; i += kRT) s_q[i / D][i % D] = __bfloat162float(qg[i]) * scale;
  const __nv_bfloat16* Kr = Kg + (size_t)j0 * D;
  const __nv_bfloat16* Vr = Vg + (size_t)j0 * D;
  if (a.kv_smem) {
    __nv_bfloat16* Ks = reinterpret_cast<__nv_bfloat16*>(dsmem + lay.Ks);
    __nv_bfloat16* Vs = reinterpret_cast<__nv_bfloat16*>(dsmem + lay.Vs);
    for (int idx = tid; idx < nr * (D / 8); idx += kRT) {
      reinterpret_cast<uint4*>(Ks)[idx] = reinterpret_cast<const uint4*>(Kr)[idx];
      reinterpret_cast<uint4*>(Vs)[idx] = reinterpret_cast<const uint4*>(Vr)[idx];
    }
    Kr = Ks;
    Vr = Vs;
  }
  if (tid == 0) {
    s_nz = 0;
    s_best[0] = s_best[1] = ~0ull;
  }
  __syncthreads();

  // ---- logits of this CTA's rows (8 lanes per row)
  for (int base = 0; base < nr; base += kRP) {
    const int j = base + rsub;
    const bool ok = j < nr;
    float kf[NC][4];
#pragma unroll
    for (int c = 0; c < NC; ++c) {
      if (ok) load4_bf16<D>(Kr + (size_t)j * D + chunk_dim<D>(q, c), kf[c]);
      else kf[c][0] = kf[c][1] = kf[c][2] = kf[c][3] = 0.f;
    }
#pragma unroll
    for (int h = 0; h < G; ++h) {
      float acc = 0.f;
#pragma unroll
      for (int c = 0; c < NC; ++c) {
        const float4 q4 = *reinterpret_cast<const float4*>(&s_q[h][chunk_dim<D>(q, c)]);
        acc = fmaf(q4.x, kf[c][0], fmaf(q4.y, kf[c][1], fmaf(q4.z, kf[c][2], fmaf(q4.w, kf[c][3], acc))));
      }
      acc = group_sum(acc);
      if (ok && q == 0) lg[h * R + j] = acc;
    }
  }
  __syncthreads();
  // softmax is shift-invariant: e_hj = exp(l_hj - M0_h) with M0_h the
  // unit's largest logit at the start.  Each CTA takes (max, sum) over its
  // rows; one cluster exchange gives M0_h and Z_h, and the CTA rescales its
  // e_hj by exp(m_h - M0_h).
  {
    float mx[G];
#pragma unroll
    for (int h = 0; h < G; ++h) mx[h] = -INFINITY;
    for (int jj = tid; jj < nr; jj += kRT)
#pragma unroll
      for (int h = 0; h < G; ++h) mx[h] = fmaxf(mx[h], lg[h * R + jj]);
#pragma unroll
    for (int h = 0; h < G; ++h) {
      mx[h] = warp_max(mx[h]);
      if (lane == 0) s_red[warp][h] = mx[h];
    }
    __syncthreads();
    if (tid < G) {
      float m = -INFINITY;
      for (int w = 0; w < kRW; ++w) m = fmaxf(m, s_red[w][tid]);
      s_M[tid] = m;
    }
    __syncthreads();
    float zs[G];
#pragma unroll
    for (int h = 0; h < G; ++h) zs[h] = 0.f;
    for (int jj = tid; jj < nr; jj += kRT)
#pragma unroll
      for (int h = 0; h < G; ++h) zs[h] += expf(lg[h * R + jj] - s_M[h]);
#pragma unroll
    for (int h = 0; h < G; ++h) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) zs[h] += __shfl_xor_sync(kFull, zs[h], o);
      if (lane == 0) s_zpart[warp][h] = zs[h];
    }
    for (int jj = len + tid; jj < a.cap; jj += kRT) alive_all[jj] = 0;
    __syncthreads();
    if (tid < G) {
      float z = 0.f;
      for (int w = 0; w < kRW; ++w) z += s_zpart[w][tid];
      s_Z[tid] = z;
    }
  }
  cluster.sync();  // every CTA's (max, sum) is published
  constexpr int P = RPW <= 8 ? 8 : 16;       // padded row count of the transposing sums
  constexpr int SH = P == 8 ? 2 : 1;         // lane l scores row l >> SH
  // Z_h lives in lane h < G of every warp as a compensated (Kahan) float,
  // decremented per eviction: value zf - zc.  Every CTA combines the
  // published partials in the same order, so all hold identical values.
  float zf = 1.f, zc = 0.f, zinv = 1.f;
  {
    __shared__ float s_Mg[G], s_Zg[G];
    if (tid < G) {  // thread h: the unit's maximum and normaliser of head h
      float mr[kCL], m = -INFINITY;
#pragma unroll
      for (int r = 0; r < kCL; ++r) {
        mr[r] = cluster.map_shared_rank(s_M, r)[tid];
        m = fmaxf(m, mr[r]);
      }
      float z = 0.f;
#pragma unroll
      for (int r = 0; r < kCL; ++r)
        if (mr[r] != -INFINITY) z += cluster.map_shared_rank(s_Z, r)[tid] * expf(mr[r] - m);
      s_Mg[tid] = m;
      s_Zg[tid] = z;
    }
    __syncthreads();
    float f[G];  // this CTA's rescale to the unit's maximum
#pragma unroll
    for (int h = 0; h < G; ++h) f[h] = s_M[h] != -INFINITY ? expf(s_M[h] - s_Mg[h]) : 0.f;
    for (int jj = tid; jj < nr; jj += kRT)
#pragma unroll
      for (int h = 0; h < G; ++h) lg[h * R + jj] = expf(lg[h * R + jj] - s_M[h]) * f[h];
    if (lane < G) {
      zf = s_Zg[lane];
      zinv = 1.f / zf;
    }
    // once no CTA reads this one's partials any more, the unit's maxima
    // replace its own (Phase 2 reads them)
    cluster.sync();
    if (tid < G) s_M[tid] = s_Mg[tid];
  }
  __syncthreads();
  // e_hj of the row this lane scores
  float ereg[G];
  {
    const int i = lane >> SH, r = warp + kRW * i;
#pragma unroll
    for (int h = 0; h < G; ++h) ereg[h] = (i < RPW && r < nr) ? lg[h * R + r] : 0.f;
  }

  // ---- registers, in the raw co-moment form S_tilde = n C (Eq. app_S_tilde):
  // y_j = S_tilde k_j of the warp's rows, the thread's share of S_tilde, the
  // means.  A Welford fold then adds (k - mu_k)(v - mu_v')^T to S_tilde and
  // ((k - mu_k) . k_j)(v - mu_v') to y_j: one FMA per element, and the clamp
  // test is |S_tilde_ab| < tau with no scaling.
  const float nf0 = static_cast<float>(n);
  float y[RPW][DPL];
  unsigned alive = 0u;
#pragma unroll
  for (int i = 0; i < RPW; ++i) {
#pragma unroll
    for (int d = 0; d < DPL; ++d) y[i][d] = 0.f;
    if (warp + kRW * i < nr) alive |= 1u << i;
  }
  if (n > 0) {
    // rows below the cache's y_len carry y_j = S_tilde k_j from the call that
    // last changed the moments (kept in the cache across calls); the others
    // (the rows appended since) are computed here, O(d^2) each
    unsigned fresh = 0u;
#pragma unroll
    for (int i = 0; i < RPW; ++i) {
      const int r = warp + kRW * i;
      if (r < nr && j0 + r < y_cur) {
        const float* src = a.Y + (row0 + j0 + r) * D + lane * DPL;
        if constexpr (DPL == 4) {
          const float4 t = *reinterpret_cast<const float4*>(src);
          y[i][0] = t.x;
          y[i][1] = t.y;
          y[i][2] = t.z;
          y[i][3] = t.w;
        } else {
          const float2 t = *reinterpret_cast<const float2*>(src);
          y[i][0] = t.x;
          y[i][1] = t.y;
        }
      } else if (r < nr) {
        fresh |= 1u << i;
      }
    }
    if (fresh != 0u) {  // warp-uniform
      for (int c = 0; c < D; ++c) {
        float cv[DPL];
        ld_vec<DPL>(Ct + (size_t)c * D + lane * DPL, cv);
#pragma unroll
        for (int i = 0; i < RPW; ++i) {
          if ((fresh >> i) & 1u) {
            const float kv = __bfloat162float(Kr[(size_t)(warp + kRW * i) * D + c]);
#pragma unroll
            for (int d = 0; d < DPL; ++d) y[i][d] = fmaf(cv[d], kv, y[i][d]);
          }
        }
      }
#pragma unroll
      for (int i = 0; i < RPW; ++i)
        if ((fresh >> i) & 1u)
#pragma unroll
          for (int d = 0; d < DPL; ++d) y[i][d] *= nf0;
    }
  }
  float creg[CJ][DPL];
#pragma unroll
  for (int jj = 0; jj < CJ; ++jj) {
    ld_vec<DPL>(Ct + (size_t)(warp + kRW * jj) * D + lane * DPL, creg[jj]);
#pragma unroll
    for (int d = 0; d < DPL; ++d) creg[jj][d] *= nf0;
  }
  float mk[DPL], mv[DPL], sdk[DPL], sdv[DPL];
#pragma unroll
  for (int d = 0; d < DPL; ++d) {
    mk[d] = s_mu_k[lane * DPL + d];
    mv[d] = s_mu_v[lane * DPL + d];
    sdk[d] = sdv[d] = 0.f;
  }
  // clamp list of the initial moments: entries with 0 < |S_tilde_ab| < tau
  const float tau = a.tau;
  if (n > 0 && tau > 0.f) {
#pragma unroll
    for (int jj = 0; jj < CJ; ++jj)
#pragma unroll
      for (int d = 0; d < DPL; ++d) {
        const float v = creg[jj][d];
        if (v != 0.f && fabsf(v) < tau) {
          const int k = atomicAdd(&s_nz, 1);
          if (k < kMaxClamp) {
            s_zidx[k] = static_cast<uint32_t>((warp + kRW * jj) * D + lane * DPL + d);
            s_zval[k] = v;
          }
        }
      }
  }
  __syncthreads();

  const int n_evict = max(0, len - a.budget);
  for (int e = 0;; ++e) {
    const int par = e & 1;
    // ---- fold the previous eviction into this thread's share of S_tilde and
    // build the clamp list: S_tilde' = S_tilde + dk dv^T
    if (e > 0) {
      const float mydk = select_n<DPL>(sdk, warp % DPL);
#pragma unroll
      for (int jj = 0; jj < CJ; ++jj) {
        const int c = warp + kRW * jj;
        const float kd = __shfl_sync(kFull, mydk, c / DPL);  // dk[c]: lane c/DPL, component warp % DPL
        bool any = false;
#pragma unroll
        for (int d = 0; d < DPL; ++d) {
          creg[jj][d] = fmaf(kd, sdv[d], creg[jj][d]);
          any |= fabsf(creg[jj][d]) < tau;
        }
        if (any) {
#pragma unroll
          for (int d = 0; d < DPL; ++d)
            if (creg[jj][d] != 0.f && fabsf(creg[jj][d]) < tau) {
              const int slot = atomicAdd(&s_nz, 1);
              if (slot < kMaxClamp) {
                s_zidx[slot] = static_cast<uint32_t>(c * D + lane * DPL + d);
                s_zval[slot] = creg[jj][d];
              }
            }
        }
      }
    }
    if (e == n_evict) break;  // uniform over the cluster
    if (tid == 0) s_best[par ^ 1] = ~0ull;  // its readers finished one iteration ago

    // ---- y_j' = y_j + (dk . k_j) dv, then the residual norms of the warp's
    // rows: r_j = v_j - mu_v - (scale / n) y_j
    const float rs = (n > 0) ? scale / static_cast<float>(n) : 0.f;
    float part[RPW];
    if (e > 0) {
#pragma unroll
      for (int i = 0; i < RPW; ++i) {
        part[i] = 0.f;
        if ((alive >> i) & 1u) {
          float kf[DPL];
          load_bf16<DPL>(Kr + (size_t)(warp + kRW * i) * D + lane * DPL, kf);
#pragma unroll
          for (int d = 0; d < DPL; ++d) part[i] = fmaf(sdk[d], kf[d], part[i]);
        }
      }
      float pv[P];
#pragma unroll
      for (int i = 0; i < P; ++i) pv[i] = i < RPW ? part[i] : 0.f;
      const float dsum = transpose_sum<P>(pv, lane);
#pragma unroll
      for (int i = 0; i < RPW; ++i) {
        const float dot = __shfl_sync(kFull, dsum, i << SH);
#pragma unroll
        for (int d = 0; d < DPL; ++d) y[i][d] = fmaf(dot, sdv[d], y[i][d]);
      }
    }
#pragma unroll
    for (int i = 0; i < RPW; ++i) {
      part[i] = 0.f;
      if ((alive >> i) & 1u) {
        float vf[DPL];
        load_bf16<DPL>(Vr + (size_t)(warp + kRW * i) * D + lane * DPL, vf);
#pragma unroll
        for (int d = 0; d < DPL; ++d) {
          const float rr = vf[d] - mv[d] - rs * y[i][d];
          part[i] = fmaf(rr, rr, part[i]);
        }
      }
    }
    // residual norms reduced so that lane l holds row l >> SH's; those lanes
    // score their row, and the warp's minimum key goes to the block minimum
    auto post_keys = [&](const float (&ss)[RPW]) {
      float pv[P];
#pragma unroll
      for (int i = 0; i < P; ++i) pv[i] = i < RPW ? ss[i] : 0.f;
      const float sum = transpose_sum<P>(pv, lane);
      float invz[G];
#pragma unroll
      for (int h = 0; h < G; ++h) invz[h] = __shfl_sync(kFull, zinv, h);
      const int i = lane >> SH;
      unsigned long long key = ~0ull;
      if ((lane & ((1 << SH) - 1)) == 0 && i < RPW && ((alive >> i) & 1u)) {
        float alpha = 0.f;
#pragma unroll
        for (int h = 0; h < G; ++h) alpha = fmaf(ereg[h], invz[h], alpha);
        const float score = alpha * sqrtf(sum);
        key = (static_cast<unsigned long long>(__float_as_uint(score)) << 32) |
              static_cast<unsigned>(j0 + warp + kRW * i);
      }
#pragma unroll
      for (int o = 16; o >= (1 << SH); o >>= 1) {
        const unsigned long long k2 = __shfl_xor_sync(kFull, key, o);
        key = k2 < key ? k2 : key;
      }
      if (lane == 0 && key != ~0ull) atomicMin(&s_best[par], key);
    };
    post_keys(part);
    __syncthreads();
    const int nz = s_nz;
    if (nz > 0) {  // uniform: clamped entries of C' change y; score again with them
      const bool direct = nz > kMaxClamp;
      if (tid == 0) s_best[par] = ~0ull;
      if (direct) {
#pragma unroll
        for (int jj = 0; jj < CJ; ++jj) st_vec<DPL>(Ct + (size_t)(warp + kRW * jj) * D + lane * DPL, creg[jj]);
      }
      __syncthreads();
#pragma unroll
      for (int i = 0; i < RPW; ++i) {
        part[i] = 0.f;
        if ((alive >> i) & 1u) {
          const int r = warp + kRW * i;
          float yc[DPL];
          if (!direct) {
#pragma unroll
            for (int d = 0; d < DPL; ++d) yc[d] = y[i][d];
            for (int z = 0; z < nz; ++z) {  // y'_a -= S_tilde_ab k_b for clamped (a, b)
              const int kb = static_cast<int>(s_zidx[z] / D), va = static_cast<int>(s_zidx[z] % D);
              if (va / DPL == lane) {
                const float corr = s_zval[z] * __bfloat162float(Kr[(size_t)r * D + kb]);
#pragma unroll
                for (int d = 0; d < DPL; ++d)
                  if (va % DPL == d) yc[d] -= corr;
              }
            }
          } else {
#pragma unroll
            for (int d = 0; d < DPL; ++d) yc[d] = 0.f;
            for (int c = 0; c < D; ++c) {
              const float kv = __bfloat162float(Kr[(size_t)r * D + c]);
              float cv[DPL];
              ld_vec<DPL>(Ct + (size_t)c * D + lane * DPL, cv);
#pragma unroll
              for (int d = 0; d < DPL; ++d) yc[d] = fmaf((fabsf(cv[d]) < tau) ? 0.f : cv[d], kv, yc[d]);
            }
          }
          float vf[DPL];
          load_bf16<DPL>(Vr + (size_t)r * D + lane * DPL, vf);
#pragma unroll
          for (int d = 0; d < DPL; ++d) {
            const float rr = vf[d] - mv[d] - rs * yc[d];
            part[i] = fmaf(rr, rr, part[i]);
          }
        }
      }
      post_keys(part);
      __syncthreads();
      if (tid == 0) s_nz = 0;  // every reader of the list is past the barrier above
    }

    // ---- warp w < 8 posts this CTA's key and candidate row into rank w's mailbox
    if (warp < kCL) {
      const unsigned long long b = s_best[par];
      const int jb = (b == ~0ull) ? -1 : static_cast<int>(b & 0xffffffffu) - j0;
      if (lane == 0) *cluster.map_shared_rank(&mail_key[par][rank], warp) = b;
      if (jb >= 0 && lane < G) *cluster.map_shared_rank(&mail_e[par][rank][lane], warp) = lg[lane * R + jb];
      if (jb >= 0 && lane < D / 4) {  // lanes 0..D/8-1 carry k, the next D/8 carry v
        const bool is_v = lane >= D / 8;
        const int i = is_v ? lane - D / 8 : lane;
        const uint4 w4 = reinterpret_cast<const uint4*>((is_v ? Vr : Kr) + (size_t)jb * D)[i];
        reinterpret_cast<uint4*>(cluster.map_shared_rank(&mail_row[par][rank][is_v ? D : 0], warp))[i] = w4;
      }
    }
    cluster.sync();

    // ---- every warp: the cluster's minimum key (ties cannot happen: rows
    // differ), by two warp-wide minimum reductions (score bits, then row)
    const unsigned long long bk = (lane < kCL) ? mail_key[par][lane] : ~0ull;
    const unsigned khi = static_cast<unsigned>(bk >> 32), klo = static_cast<unsigned>(bk);
    const unsigned mhi = __reduce_min_sync(kFull, khi);
    const unsigned mlo = __reduce_min_sync(kFull, khi == mhi ? klo : 0xffffffffu);
    const int src = __ffs(__ballot_sync(kFull, khi == mhi && klo == mlo)) - 1;
    const int js = (mhi == 0xffffffffu && mlo == 0xffffffffu) ? -1 : static_cast<int>(mlo);
    if (js < 0) {  // uniform: every rank read the same keys
      if (rank == 0 && tid == 0) record_error(a.ws, MKV_ERR_INVALID_ARG, u);
      break;
    }
    // Welford fold of the evicted row for this lane's dims (Eq. app_update)
    {
      const float inv = 1.f / static_cast<float>(n + 1);
      float kx[DPL], vx[DPL];
      load_bf16<DPL>(&mail_row[par][src][lane * DPL], kx);
      load_bf16<DPL>(&mail_row[par][src][D + lane * DPL], vx);
#pragma unroll
      for (int d = 0; d < DPL; ++d) {
        const float dk = kx[d] - mk[d];
        mk[d] = fmaf(dk, inv, mk[d]);
        mv[d] = fmaf(vx[d] - mv[d], inv, mv[d]);
        sdk[d] = dk;
        sdv[d] = vx[d] - mv[d];
      }
      n += 1;
    }
    const int jr = js - j0;
    if (jr >= 0 && jr < nr && jr % kRW == warp) alive &= ~(1u << (jr / kRW));
    if (lane < G) {  // compensated Z_h -= e_h,js
      const float yk = -mail_e[par][src][lane] - zc;
      const float tk = zf + yk;
      zc = (tk - zf) - yk;
      zf = tk;
      zinv = 1.f / zf;
    }
  }

  // ---- state back to shared memory: survivors, C (transposed), means
#pragma unroll
  for (int i = 0; i < RPW; ++i)
    if (lane == 0 && warp + kRW * i < nr) alive_all[j0 + warp + kRW * i] = (alive >> i) & 1u;
#pragma unroll
  for (int jj = 0; jj < CJ; ++jj) {
    float cv[DPL];
#pragma unroll
    for (int d = 0; d < DPL; ++d) cv[d] = n > 0 ? creg[jj][d] / static_cast<float>(n) : 0.f;
    st_vec<DPL>(Ct + (size_t)(warp + kRW * jj) * D + lane * DPL, cv);
  }
  if (warp == 0) {
#pragma unroll
    for (int d = 0; d < DPL; ++d) {
      s_mu_k[lane * DPL + d] = mk[d];
      s_mu_v[lane * DPL + d] = mv[d];
    }
  }
  __syncthreads();
  const uint8_t* alv = alive_all + j0;

  // ---- ordered compaction across the cluster through the staging buffer
  {
    int cnt = 0;
    for (int r = tid; r < nr; r += kRT) cnt += alv[r];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(kFull, cnt, o);
    if (lane == 0) s_red[warp][0] = static_cast<float>(cnt);
    __syncthreads();
    if (tid == 0) {
      int c = 0;
      for (int w = 0; w < kRW; ++w) c += static_cast<int>(s_red[w][0]);
      ex_cnt = c;
    }
  }
  cluster.sync();
  int base = 0;
  for (int r = 0; r < rank; ++r) base += *cluster.map_shared_rank(&ex_cnt, r);
  const int mine = ex_cnt;
  if (a.Y != nullptr && a.y_len != nullptr) {
    // the loop left the last eviction folded into S_tilde but not yet into
    // y: y_j += (dk . k_j) dv for the surviving rows, as in the loop
    {
      float part[RPW];
#pragma unroll
      for (int i = 0; i < RPW; ++i) {
        part[i] = 0.f;
        if ((alive >> i) & 1u) {
          float kf[DPL];
          load_bf16<DPL>(Kr + (size_t)(warp + kRW * i) * D + lane * DPL, kf);
#pragma unroll
          for (int d = 0; d < DPL; ++d) part[i] = fmaf(sdk[d], kf[d], part[i]);
        }
      }
      float pv[P];
#pragma unroll
      for (int i = 0; i < P; ++i) pv[i] = i < RPW ? part[i] : 0.f;
      const float dsum = transpose_sum<P>(pv, lane);
#pragma unroll
      for (int i = 0; i < RPW; ++i) {
        const float dot = __shfl_sync(kFull, dsum, i << SH);
#pragma unroll
        for (int d = 0; d < DPL; ++d) y[i][d] = fmaf(dot, sdv[d], y[i][d]);
      }
    }
    // y_j of the surviving rows to their compacted rows: each warp writes its
    // own rows' registers (every read of the y rows was in the set-up, before
    // the cluster barriers of the loop)
#pragma unroll
    for (int i = 0; i < RPW; ++i) {
      const int r = warp + kRW * i;
      if (r < nr && ((alive >> i) & 1u)) {  // warp-uniform
        int before = 0;  // survivors of this CTA ahead of row r
        for (int c0 = 0; c0 < r; c0 += 32)
          before += __popc(__ballot_sync(kFull, c0 + lane < r && alv[c0 + lane]));
        float* dst = a.Y + (row0 + base + before) * D + lane * DPL;
        if constexpr (DPL == 4) *reinterpret_cast<float4*>(dst) = make_float4(y[i][0], y[i][1], y[i][2], y[i][3]);
        else *reinterpret_cast<float2*>(dst) = make_float2(y[i][0], y[i][1]);
      }
    }
    if (rank == 0 && tid == 0) a.y_len[u] = a.budget;  // ordered after the other CTAs' writes by the kernel end
  }
  uint8_t* st = static_cast<uint8_t*>(a.stage) + (size_t)u * stage_stride(a.cap, D);
  __nv_bfloat16* SK = reinterpret_cast<__nv_bfloat16*>(st);
  __nv_bfloat16* SV = SK + (size_t)a.cap * D;
  int32_t* SP = reinterpret_cast<int32_t*>(SV + (size_t)a.cap * D);
  for (int c0 = 0; c0 < nr; c0 += 32) {
    const bool al = (c0 + lane < nr) && alv[c0 + lane];
    const unsigned m = __ballot_sync(kFull, al);
    int before = 0;  // survivors in earlier chunks
    for (int c1 = 0; c1 < c0; c1 += 32) {
      const bool a1 = (c1 + lane < nr) && alv[c1 + lane];
      before += __popc(__ballot_sync(kFull, a1));
    }
    for (int bit = warp; bit < 32; bit += kRW) {  // warp w moves rows c0 + w, c0 + w + 16
      if ((m >> bit) & 1u) {
        const int r = c0 + bit;
        const int dst = base + before + __popc(m & ((1u << bit) - 1u));
        for (int i = lane; i < D / 8; i += 32) {
          reinterpret_cast<uint4*>(SK + (size_t)dst * D)[i] = reinterpret_cast<const uint4*>(Kr + (size_t)r * D)[i];
          reinterpret_cast<uint4*>(SV + (size_t)dst * D)[i] = reinterpret_cast<const uint4*>(Vr + (size_t)r * D)[i];
        }
        if (lane == 0) SP[dst] = Pg[j0 + r];
      }
    }
  }
  __threadfence();
  cluster.sync();
  for (int idx = tid; idx < mine * (D / 8); idx += kRT) {
    const int row = base + idx / (D / 8), i = idx % (D / 8);
    reinterpret_cast<uint4*>(Kg + (size_t)row * D)[i] = reinterpret_cast<const uint4*>(SK + (size_t)row * D)[i];
    reinterpret_cast<uint4*>(Vg + (size_t)row * D)[i] = reinterpret_cast<const uint4*>(SV + (size_t)row * D)[i];
  }
  for (int r = tid; r < mine; r += kRT) Pg[base + r] = SP[base + r];
  {  // C back to global, its 32 x 32 tiles shared out over the cluster's CTAs
    float* tb = s_tile[warp % kTWR];
    for (int t = rank + kCL * warp; warp < kTWR && t < (D / 32) * (D / 32); t += kCL * kTWR) {
      const int c0 = (t / (D / 32)) * 32, r0 = (t % (D / 32)) * 32;
      for (int i = 0; i < 32; ++i) tb[i * 33 + lane] = Ct[(size_t)(c0 + i) * D + r0 + lane];
      __syncwarp();
      for (int i = 0; i < 32; ++i) a.C[(size_t)u * D * D + (size_t)(r0 + i) * D + c0 + lane] = tb[lane * 33 + i];
      __syncwarp();
    }
  }
  if (rank == 0) {
    for (int i = tid; i < D; i += kRT) {
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
  const size_t with_kv = ClusterLayout<D, G>(R, cap, 1).total;
  if (with_kv <= kSmemBudget) {
    *kv = 1;
    return with_kv;
  }
  *kv = 0;
  return ClusterLayout<D, G>(R, cap, 0).total;
}

template <int D, int G, int RPW>
cudaError_t launch_reg(EvictArgs a, cudaStream_t stream) {
  a.rows_max = (a.cap + kCL - 1) / kCL;
  a.kv_smem = 1;
  size_t smem = RegLayout<D, G>(a.rows_max, a.cap, 1).total;
  if (smem > kSmemBudget) {
    a.kv_smem = 0;
    smem = RegLayout<D, G>(a.rows_max, a.cap, 0).total;
  }
  cudaError_t e = cudaFuncSetAttribute(evict_reg_kernel<D, G, RPW>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  evict_reg_kernel<D, G, RPW><<<a.batch * a.n_kv * kCL, kRT, smem, stream>>>(a);
  return cudaGetLastError();
}

template <int D, int G>
cudaError_t launch_dg(const EvictArgs& a0, cudaStream_t stream) {
  EvictArgs a = a0;
  // rows of one CTA's slice at most; warps of the register kernel hold 5 or 9 each
  const int slice = (a.cap + kCL - 1) / kCL;
  if (slice <= kRW * 5) return launch_reg<D, G, 5>(a, stream);
  if (slice <= kRW * 9) return launch_reg<D, G, 9>(a, stream);
  int kv = 0;
  const size_t csm = cluster_smem<D, G>(a.cap, &kv);
  if (csm <= kSmemBudget) {
    a.rows_max = (a.cap + kCL - 1) / kCL;
    a.kv_smem = kv;
    cudaError_t e = cudaFuncSetAttribute(evict_cluster_kernel<D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(csm));
    if (e != cudaSuccess) return e;
    evict_cluster_kernel<D, G><<<a.batch * a.n_kv * kCL, kCT, csm, stream>>>(a);
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
