// Decode step: retained-cache attention merged with the moment correction
// (Algorithm 1 Phase 2; Eqs. jensen, fhat, fused; log-domain merge of App. C.2).
//
// Grid (S, h_kv, b): every CTA serves all G query heads of one KV head
// (GQA grouping, so K/V rows are read once per unit) over one contiguous
// split of the retained rows.  Rows stream from HBM through a 4-stage ring of
// shared-memory tiles filled by 1-D bulk copies (TMA engine, mbarrier
// completion); compute is an online softmax per head.  The moment term
// S_tilde q / (n sqrt d) is spread over the same CTAs: CTA s computes rows
// [s*D/S, ...) of C'q for all G heads, so C (64 KB fp32 at d=128) is read once
// per unit, concurrently with the K/V stream.  The last CTA of a unit to
// finish (atomic ticket, no waiting) merges the S partial (m, l, o) states and
// the moment pseudo-partial (log n + scale q.mu_k, f_hat_E) with a
// log-sum-exp and writes the output; it also performs the append.
#include "common.cuh"
#include "kernels.h"

namespace mkv {

namespace {

constexpr int kThreads = 128;  // 4 warps, 8 tokens of each tile per warp
constexpr int kStages = 4;
constexpr int kTT = kDecodeTile;
constexpr unsigned kFull = 0xffffffffu;

// Butterfly transpose-reduction: each lane holds N partial sums (N = 8*G,
// value index = token*G + head); afterwards lane l holds the full sums of
// value indices [l*R, l*R+R) with R = max(1, N/32) (for N < 32 lanes that
// differ only in the low bits hold copies: index = l >> log2(32/N)).
template <int N>
__device__ __forceinline__ void transpose_reduce(float (&v)[N], int lane) {
#pragma unroll
  for (int k = 0; k < 5; ++k) {
    const int off = 16 >> k;
    const int half = (N >> k) / 2;
    if (half >= 1) {
      const bool upper = (lane & off) != 0;
#pragma unroll
      for (int i = 0; i < (N >> (k + 1)); ++i) {
        const float send = upper ? v[i] : v[i + (N >> (k + 1))];
        const float keep = upper ? v[i + (N >> (k + 1))] : v[i];
        v[i] = keep + __shfl_xor_sync(kFull, send, off);
      }
    } else {
      v[0] += __shfl_xor_sync(kFull, v[0], off);
    }
  }
}

// Lane that holds (token j, head h) after transpose_reduce, and which of its
// R values it is.
template <int G>
__device__ __forceinline__ int src_lane(int j, int h) {
  if constexpr (G == 1) return j << 2;
  else if constexpr (G == 2) return (j << 2) | (h << 1);
  else if constexpr (G == 4) return (j << 2) | h;
  else return (j << 2) | (h >> 1);
}

template <int G>
__device__ __forceinline__ int my_head(int lane, int r) {
  if constexpr (G == 1) return 0;
  else if constexpr (G == 2) return (lane >> 1) & 1;
  else if constexpr (G == 4) return lane & 3;
  else return ((lane & 3) << 1) | r;
}

template <int D, int G>
struct WarpState {
  static constexpr int DPL = D / 32;
  float m[G];  // running max, log2 domain, replicated across lanes
  float l[G];  // running sum, replicated
  float o[G][DPL];
};

// Process up to 8 rows (this warp's slice of a tile) of K/V in shared memory.
template <int D, int G>
__device__ __forceinline__ void process_rows(WarpState<D, G>& st, const float (&qr)[G][D / 32],
                                             const __nv_bfloat16* tK, const __nv_bfloat16* tV,
                                             int row0, int rows, int lane) {
  constexpr int DPL = D / 32;
  constexpr int N = 8 * G;
  constexpr int R = (N >= 32) ? N / 32 : 1;
  float v[N];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    float kf[DPL];
    if (row0 + j < rows) {
      load_bf16<DPL>(tK + (row0 + j) * D + lane * DPL, kf);
    } else {
#pragma unroll
      for (int i = 0; i < DPL; ++i) kf[i] = 0.f;
    }
#pragma unroll
    for (int h = 0; h < G; ++h) {
      float acc = 0.f;
#pragma unroll
      for (int i = 0; i < DPL; ++i) acc = fmaf(qr[h][i], kf[i], acc);
      v[j * G + h] = acc;
    }
  }
  transpose_reduce<N>(v, lane);

  const int j = lane >> 2;
  const bool valid = (row0 + j) < rows;
  float sc[R], tmax[R];
#pragma unroll
  for (int r = 0; r < R; ++r) {
    sc[r] = valid ? v[r] : -INFINITY;
    tmax[r] = sc[r];
#pragma unroll
    for (int off = 4; off <= 16; off <<= 1) tmax[r] = fmaxf(tmax[r], __shfl_xor_sync(kFull, tmax[r], off));
  }
  // every lane learns every head's new running max and rescale factor
  float mnew[G], alpha[G];
#pragma unroll
  for (int h = 0; h < G; ++h) {
    const float tm = __shfl_sync(kFull, tmax[(G == 8) ? (h & 1) : 0], src_lane<G>(0, h));
    mnew[h] = fmaxf(st.m[h], tm);
    alpha[h] = (mnew[h] == -INFINITY) ? 1.f : fast_exp2(st.m[h] - mnew[h]);
  }
  float p[R], ls[R];
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int hh = my_head<G>(lane, r);
    float mm = 0.f;
#pragma unroll
    for (int h = 0; h < G; ++h) mm = (h == hh) ? mnew[h] : mm;
    p[r] = valid ? fast_exp2(sc[r] - mm) : 0.f;
    ls[r] = p[r];
#pragma unroll
    for (int off = 4; off <= 16; off <<= 1) ls[r] += __shfl_xor_sync(kFull, ls[r], off);
  }
#pragma unroll
  for (int h = 0; h < G; ++h) {
    const float lt = __shfl_sync(kFull, ls[(G == 8) ? (h & 1) : 0], src_lane<G>(0, h));
    st.l[h] = st.l[h] * alpha[h] + lt;
    st.m[h] = mnew[h];
#pragma unroll
    for (int i = 0; i < DPL; ++i) st.o[h][i] *= alpha[h];
  }
#pragma unroll
  for (int jj = 0; jj < 8; ++jj) {
    if (row0 + jj >= rows) break;  // warp-uniform
    float vf[DPL];
    load_bf16<DPL>(tV + (row0 + jj) * D + lane * DPL, vf);
#pragma unroll
    for (int h = 0; h < G; ++h) {
      const float pj = __shfl_sync(kFull, p[(G == 8) ? (h & 1) : 0], src_lane<G>(jj, h));
#pragma unroll
      for (int i = 0; i < DPL; ++i) st.o[h][i] = fmaf(pj, vf[i], st.o[h][i]);
    }
  }
}

template <int D, int G>
__global__ void __launch_bounds__(kThreads) decode_kernel(const DecodeArgs a) {
  constexpr int DPL = D / 32;
  constexpr int PS = D + 4;  // partial record: o[D], m (log2 domain), l
  extern __shared__ __align__(128) uint8_t dsmem[];
  __nv_bfloat16* sK = reinterpret_cast<__nv_bfloat16*>(dsmem);
  __nv_bfloat16* sV = sK + kStages * kTT * D;
  __nv_bfloat16* sNew = sV + kStages * kTT * D;  // [2][D]: new k, new v
  __shared__ float sQ[G * D];                      // q * scale * log2(e)
  __shared__ float sSbar[G];
  __shared__ float sM[G], sL[G];
  __shared__ __align__(8) uint64_t bars[kStages];
  __shared__ int sTicket;

  const int s = blockIdx.x, kv = blockIdx.y, b = blockIdx.z;
  const int u = b * a.n_kv + kv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  int len0 = a.len[u];
  if (len0 < 0 || len0 > a.cap) {  // corrupt cache state: never read past the slab
    if (tid == 0 && s == 0) record_error(a.ws, MKV_ERR_CAPACITY, u);
    len0 = len0 < 0 ? 0 : a.cap;
  }
  const bool has_new = a.k_new != nullptr;
  const int L = len0 + (has_new ? 1 : 0);
  const int n_e = (a.correction != 0 && a.n != nullptr) ? a.n[u] : 0;
  const bool use_m = n_e > 0;
  const float scale = rsqrtf(static_cast<float>(D));

  const int tiles_total = (L + kTT - 1) / kTT;
  const int tiles_per = (tiles_total + a.S - 1) / a.S;
  const int t_begin = min(L, s * tiles_per * kTT);
  const int t_end = min(L, t_begin + tiles_per * kTT);
  const int n_cached = max(0, min(t_end, len0) - t_begin);
  const bool own_new = has_new && t_begin <= len0 && len0 < t_end;
  const int n_tiles = (n_cached + kTT - 1) / kTT;

  const __nv_bfloat16* Kg = reinterpret_cast<const __nv_bfloat16*>(a.K) + ((size_t)u * a.cap + t_begin) * D;
  const __nv_bfloat16* Vg = reinterpret_cast<const __nv_bfloat16*>(a.V) + ((size_t)u * a.cap + t_begin) * D;

  auto issue = [&](int it) {
    const int st = it % kStages;
    const int rows = min(kTT, n_cached - it * kTT);
    const uint32_t bytes = static_cast<uint32_t>(rows) * D * 2u;
    mbar_arrive_expect_tx(&bars[st], 2u * bytes);
    bulk_g2s(sK + st * kTT * D, Kg + (size_t)it * kTT * D, bytes, &bars[st]);
    bulk_g2s(sV + st * kTT * D, Vg + (size_t)it * kTT * D, bytes, &bars[st]);
  };

  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) mbar_init(&bars[i], 1);
    mbar_fence_init();
  }
  __syncthreads();
  if (tid == 0) {
    for (int i = 0; i < min(kStages, n_tiles); ++i) issue(i);
  }

  const __nv_bfloat16* qg = reinterpret_cast<const __nv_bfloat16*>(a.q) + ((size_t)u * G) * D;
  for (int i = tid; i < G * D; i += kThreads) sQ[i] = __bfloat162float(qg[i]) * (scale * kLog2e);
  __syncthreads();

  // ---- moment rows: f_hat_E[h][row] = mu_v[row] + scale * sum_c C'[row][c] q_h[c]
  // (each warp keeps RB rows' loads in flight before reducing them)
  if (use_m && a.order == 1) {
    constexpr int RB = 4;
    const int rpc = (D + a.S - 1) / a.S;
    const int r0 = s * rpc, r1 = min(D, r0 + rpc);
    const float tau = a.tau;
    const float nf = static_cast<float>(n_e);
    for (int base = r0 + warp; base < r1; base += 4 * RB) {
      float cv[RB][DPL];
      float mv[RB];
#pragma unroll
      for (int k = 0; k < RB; ++k) {
        const int row = base + 4 * k;
        mv[k] = 0.f;
#pragma unroll
        for (int i = 0; i < DPL; ++i) cv[k][i] = 0.f;
        if (row < r1) {
          const float* Crow = a.C + ((size_t)u * D + row) * D + lane * DPL;
          if constexpr (DPL == 4) {
            const float4 t = __ldg(reinterpret_cast<const float4*>(Crow));
            cv[k][0] = t.x; cv[k][1] = t.y; cv[k][2] = t.z; cv[k][3] = t.w;
          } else {
            const float2 t = __ldg(reinterpret_cast<const float2*>(Crow));
            cv[k][0] = t.x; cv[k][1] = t.y;
          }
          if (lane == 0) mv[k] = __ldg(a.mu_v + (size_t)u * D + row);
        }
      }
#pragma unroll
      for (int k = 0; k < RB; ++k) {
        const int row = base + 4 * k;
        if (row >= r1) break;  // warp-uniform
#pragma unroll
        for (int i = 0; i < DPL; ++i) cv[k][i] = (fabsf(cv[k][i] * nf) < tau) ? 0.f : cv[k][i];
        float acc[G];
#pragma unroll
        for (int h = 0; h < G; ++h) {
          acc[h] = 0.f;
#pragma unroll
          for (int i = 0; i < DPL; ++i) acc[h] = fmaf(cv[k][i], sQ[h * D + lane * DPL + i], acc[h]);
          acc[h] = warp_sum(acc[h]);
        }
        if (lane == 0) {
#pragma unroll
          for (int h = 0; h < G; ++h) a.fhat[((size_t)u * G + h) * D + row] = mv[k] + acc[h] * (1.f / kLog2e);
        }
      }
    }
  }

  // ---- retained rows
  WarpState<D, G> st;
  float qr[G][DPL];
#pragma unroll
  for (int h = 0; h < G; ++h) {
    st.m[h] = -INFINITY;
    st.l[h] = 0.f;
#pragma unroll
    for (int i = 0; i < DPL; ++i) {
      st.o[h][i] = 0.f;
      qr[h][i] = sQ[h * D + lane * DPL + i];
    }
  }
  bool ok = true;
  int it = 0;
  for (; it < n_tiles; ++it) {
    const int stg = it % kStages;
    const bool got = mbar_wait(&bars[stg], (it / kStages) & 1);
    if (!__syncthreads_and(got)) {
      ok = false;
      break;
    }
    const int rows = min(kTT, n_cached - it * kTT);
    process_rows<D, G>(st, qr, sK + stg * kTT * D, sV + stg * kTT * D, warp * 8, rows, lane);
    __syncthreads();
    if (tid == 0 && it + kStages < n_tiles) issue(it + kStages);
  }
  if (!ok) {
    if (tid == 0) {
      record_error(a.ws, MKV_ERR_TIMEOUT, u);
      // drain the copies still owed to this CTA before its shared memory is released
      for (int j = it; j < min(n_tiles, it + kStages); ++j) (void)mbar_wait(&bars[j % kStages], (j / kStages) & 1);
    }
    __syncthreads();
#pragma unroll
    for (int h = 0; h < G; ++h) {
      st.m[h] = -INFINITY;
      st.l[h] = 0.f;
    }
  }
  if (own_new) {
    const __nv_bfloat16* kn = reinterpret_cast<const __nv_bfloat16*>(a.k_new) + (size_t)u * D;
    const __nv_bfloat16* vn = reinterpret_cast<const __nv_bfloat16*>(a.v_new) + (size_t)u * D;
    for (int i = tid; i < D; i += kThreads) {
      sNew[i] = kn[i];
      sNew[D + i] = vn[i];
    }
    __syncthreads();
    if (warp == 0) process_rows<D, G>(st, qr, sNew, sNew + D, 0, 1, lane);
  }

  // ---- merge the 4 warps into this CTA's partial record (through the free tile ring)
  float* sRed = reinterpret_cast<float*>(dsmem);  // [4][G][D + 2]
  __syncthreads();
#pragma unroll
  for (int h = 0; h < G; ++h) {
#pragma unroll
    for (int i = 0; i < DPL; ++i) sRed[(warp * G + h) * (D + 2) + lane * DPL + i] = st.o[h][i];
    if (lane == 0) {
      sRed[(warp * G + h) * (D + 2) + D] = st.m[h];
      sRed[(warp * G + h) * (D + 2) + D + 1] = st.l[h];
    }
  }
  __syncthreads();
  float* part = a.partial + ((size_t)u * a.S + s) * G * PS;
  for (int idx = tid; idx < G * D; idx += kThreads) {
    const int h = idx / D, dd = idx % D;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 4; ++w) M = fmaxf(M, sRed[(w * G + h) * (D + 2) + D]);
    float o = 0.f, l = 0.f;
    if (M != -INFINITY) {
#pragma unroll
      for (int w = 0; w < 4; ++w) {
        const float* rw = sRed + (w * G + h) * (D + 2);
        const float f = fast_exp2(rw[D] - M);
        o = fmaf(f, rw[dd], o);
        l = fmaf(f, rw[D + 1], l);
      }
    }
    part[h * PS + dd] = o;
    if (dd == 0) {
      part[h * PS + D] = M;
      part[h * PS + D + 1] = l;
    }
  }

  // ---- ticket: the last CTA of this unit merges everything
  __threadfence();
  __syncthreads();
  if (tid == 0) sTicket = static_cast<int>(atomicAdd(&a.counters[u], 1u));
  __syncthreads();
  if (sTicket != a.S - 1) return;
  __threadfence();
  if (tid == 0) a.counters[u] = 0u;

  if (use_m) {
    for (int h = warp; h < G; h += 4) {
      float acc = 0.f;
      for (int c = lane; c < D; c += 32) acc = fmaf(sQ[h * D + c], a.mu_k[(size_t)u * D + c], acc);
      acc = warp_sum(acc);
      if (lane == 0) sSbar[h] = acc * (1.f / kLog2e);  // scale * q . mu_k
    }
  }
  __syncthreads();

  // combine the S partial records: per-(split, head) weights in shared
  // memory, then each thread accumulates 4 output dims with all loads in flight
  const float* pu = a.partial + (size_t)u * a.S * G * PS;
  float* sW = reinterpret_cast<float*>(dsmem);  // [S][G] max, then weight
  float* sLs = sW + a.S * G;                    // [S][G] sums
  __syncthreads();
  for (int i = tid; i < a.S * G; i += kThreads) {
    sW[i] = __ldcg(pu + (size_t)i * PS + D);
    sLs[i] = __ldcg(pu + (size_t)i * PS + D + 1);
  }
  __syncthreads();
  if (tid < G) {
    float M = -INFINITY;
    for (int sp = 0; sp < a.S; ++sp)
      if (sLs[sp * G + tid] > 0.f) M = fmaxf(M, sW[sp * G + tid]);
    float l = 0.f;
    if (M != -INFINITY)
      for (int sp = 0; sp < a.S; ++sp)
        if (sLs[sp * G + tid] > 0.f) l = fmaf(sLs[sp * G + tid], fast_exp2(sW[sp * G + tid] - M), l);
    sM[tid] = M;
    sL[tid] = l;
  }
  __syncthreads();
  for (int i = tid; i < a.S * G; i += kThreads) {
    const float M = sM[i % G];
    sW[i] = (sLs[i] > 0.f && M != -INFINITY) ? fast_exp2(sW[i] - M) : 0.f;
  }
  __syncthreads();
  for (int slot = tid; slot < G * (D / 4); slot += kThreads) {
    const int h = slot / (D / 4), d0 = (slot % (D / 4)) * 4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
    for (int sp = 0; sp < a.S; ++sp) {
      const float w = sW[sp * G + h];
      const float4 o = __ldcg(reinterpret_cast<const float4*>(pu + ((size_t)sp * G + h) * PS + d0));
      acc.x = fmaf(w, o.x, acc.x);
      acc.y = fmaf(w, o.y, acc.y);
      acc.z = fmaf(w, o.z, acc.z);
      acc.w = fmaf(w, o.w, acc.w);
    }
    const float l = sL[h];
    const bool have_r = l > 0.f;
    const float aR = have_r ? sM[h] * kLn2 + logf(l) : -INFINITY;
    const float inv_l = have_r ? 1.f / l : 0.f;
    const float oR[4] = {acc.x * inv_l, acc.y * inv_l, acc.z * inv_l, acc.w * inv_l};
    float res[4], lse = aR;
    if (use_m) {
      const float e = logf(static_cast<float>(n_e)) + sSbar[h];
      float fh[4];
#pragma unroll
      for (int k = 0; k < 4; ++k)
        fh[k] = (a.order == 1) ? __ldcg(a.fhat + ((size_t)u * G + h) * D + d0 + k) : a.mu_v[(size_t)u * D + d0 + k];
      if (have_r) {
        const float top = fmaxf(aR, e);
        const float wr = expf(aR - top), we = expf(e - top);
        const float wR = wr / (wr + we);
#pragma unroll
        for (int k = 0; k < 4; ++k) res[k] = wR * oR[k] + (1.f - wR) * fh[k];
        lse = top + logf(wr + we);
      } else {
#pragma unroll
        for (int k = 0; k < 4; ++k) res[k] = fh[k];
        lse = e;
      }
    } else {
      if (!have_r && d0 == 0 && h == 0) record_error(a.ws, MKV_ERR_INVALID_ARG, u);
#pragma unroll
      for (int k = 0; k < 4; ++k) res[k] = oR[k];
    }
    *reinterpret_cast<float4*>(a.out + ((size_t)u * G + h) * D + d0) = make_float4(res[0], res[1], res[2], res[3]);
    if (a.lse != nullptr && d0 == 0) a.lse[(size_t)u * G + h] = lse;
  }

  if (has_new) {
    if (len0 + 1 > a.cap) {
      if (tid == 0) record_error(a.ws, MKV_ERR_CAPACITY, u);
    } else {
      const __nv_bfloat16* kn = reinterpret_cast<const __nv_bfloat16*>(a.k_new) + (size_t)u * D;
      const __nv_bfloat16* vn = reinterpret_cast<const __nv_bfloat16*>(a.v_new) + (size_t)u * D;
      __nv_bfloat16* Kd = reinterpret_cast<__nv_bfloat16*>(a.K) + ((size_t)u * a.cap + len0) * D;
      __nv_bfloat16* Vd = reinterpret_cast<__nv_bfloat16*>(a.V) + ((size_t)u * a.cap + len0) * D;
      for (int i = tid; i < D; i += kThreads) {
        Kd[i] = kn[i];
        Vd[i] = vn[i];
      }
      if (tid == 0) {
        a.pos[(size_t)u * a.cap + len0] = a.seen[u];
        a.seen[u] = a.seen[u] + 1;
        a.len[u] = len0 + 1;
      }
    }
  }
}

template <int D, int G>
cudaError_t launch_dg(const DecodeArgs& a, cudaStream_t stream) {
  const size_t smem = (size_t)(2 * kStages * kTT * D + 2 * D) * sizeof(__nv_bfloat16);
  // per-device function attribute; setting it again is harmless
  cudaError_t e = cudaFuncSetAttribute(decode_kernel<D, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  dim3 grid(a.S, a.n_kv, a.batch);
  decode_kernel<D, G><<<grid, kThreads, smem, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace

int decode_splits(const mkv_geom& g, int32_t capacity, int num_sms) {
  const long units = (long)g.batch * g.n_kv_heads;
  const long tiles = ((long)capacity + 1 + kTT - 1) / kTT;
  long S = (8L * num_sms + units - 1) / units;
  if (S > tiles) S = tiles;
  if (S > 64) S = 64;
  if (S < 1) S = 1;
  return static_cast<int>(S);
}

size_t decode_workspace_bytes(const mkv_geom& g, int32_t capacity, int num_sms) {
  const size_t units = (size_t)g.batch * g.n_kv_heads;
  const int S = decode_splits(g, capacity, num_sms);
  size_t off = kHeaderBytes;
  off += align_up(units * sizeof(uint32_t), 256);
  off += align_up(units * S * g.group * (g.head_dim + 4) * sizeof(float), 256);
  off += align_up(units * g.group * g.head_dim * sizeof(float), 256);
  return off;
}

void decode_carve(DecodeArgs& a, const mkv_geom& g, int32_t capacity, int num_sms, void* ws) {
  const size_t units = (size_t)g.batch * g.n_kv_heads;
  const int S = decode_splits(g, capacity, num_sms);
  uint8_t* p = static_cast<uint8_t*>(ws);
  a.ws = ws;
  size_t off = kHeaderBytes;
  a.counters = reinterpret_cast<uint32_t*>(p + off);
  off += align_up(units * sizeof(uint32_t), 256);
  a.partial = reinterpret_cast<float*>(p + off);
  off += align_up(units * S * g.group * (g.head_dim + 4) * sizeof(float), 256);
  a.fhat = reinterpret_cast<float*>(p + off);
  a.S = S;
}

size_t decode_workspace_bytes_splits(const mkv_geom& g, int S) {
  const size_t units = (size_t)g.batch * g.n_kv_heads;
  size_t off = kHeaderBytes;
  off += align_up(units * sizeof(uint32_t), 256);
  off += align_up(units * S * g.group * (g.head_dim + 4) * sizeof(float), 256);
  off += align_up(units * g.group * g.head_dim * sizeof(float), 256);
  return off;
}

void decode_carve_splits(DecodeArgs& a, const mkv_geom& g, int S, void* ws) {
  const size_t units = (size_t)g.batch * g.n_kv_heads;
  uint8_t* p = static_cast<uint8_t*>(ws);
  a.ws = ws;
  size_t off = kHeaderBytes;
  a.counters = reinterpret_cast<uint32_t*>(p + off);
  off += align_up(units * sizeof(uint32_t), 256);
  a.partial = reinterpret_cast<float*>(p + off);
  off += align_up(units * S * g.group * (g.head_dim + 4) * sizeof(float), 256);
  a.fhat = reinterpret_cast<float*>(p + off);
  a.S = S;
}

cudaError_t launch_decode(const DecodeArgs& a, int head_dim, int group, cudaStream_t stream) {
#define MKV_DECODE_CASE(D, G) \
  if (head_dim == D && group == G) return launch_dg<D, G>(a, stream);
  MKV_DECODE_CASE(128, 1)
  MKV_DECODE_CASE(128, 2)
  MKV_DECODE_CASE(128, 4)
  MKV_DECODE_CASE(128, 8)
  MKV_DECODE_CASE(64, 1)
  MKV_DECODE_CASE(64, 2)
  MKV_DECODE_CASE(64, 4)
  MKV_DECODE_CASE(64, 8)
#undef MKV_DECODE_CASE
  return cudaErrorInvalidValue;
}

}  // namespace mkv
