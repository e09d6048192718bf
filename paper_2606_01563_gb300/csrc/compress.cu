// Prefill compression (Sec. 5.1 SnapKV protocol with the moment filter of
// Sec. 4.2, read as two data-parallel selection stages).
//
// Launch sequence per call (all on one stream):
//   stats    (chunk, unit)  window-row online (max, sum) of the causal logits
//                           l = scale q . k, and the chunk's centred moments
//                           (n_c, mean k, mean v, co-moment M_c = sum (v-mv)(k-mk)^T)
//   scores   (chunk, unit)  s_t = sum over rows of exp(l - m_row) / l_row,
//                           pooled into aligned chunks of `pool` tokens
//   select   (unit)         R0 = protected + top-k(s)   (radix select, ties
//                           to the lower position), mean k/v of R0
//   moments  (rows, unit)   moments of E0 = all \ R0: multi-way Chan merge of
//                           the chunk moments minus R0's own centred moments
//   residual (chunk, unit)  score2_t = s_t ||v_t - mu_v0 - scale C0' k_t||
//   select   (unit)         R = protected + top-k(score2)
//   moments  (rows, unit)   moments of E = all \ R -> caller's mkv_moments
//   gather   (rows, unit)   retained rows of R, ascending, -> caller's cache
#include "common.cuh"
#include "kernels.h"

namespace mkv {

namespace {

constexpr int kTT = 32;  // tokens per tile (one per lane)
constexpr unsigned kFull = 0xffffffffu;

struct Layout {
  int D, G, W, RW;  // head dim, group, window, window rows = G*W
  int T, B;
  int units, n_chunks, chunk;
  size_t rec;  // floats per chunk-moment record: 4 + 2D + D*D (padded)
  // carved pointers
  float* rowpart;   // [units][n_chunks][RW][2]
  float* mpart;     // [units][n_chunks][rec]
  float* s;         // [units][T]
  float* s2;        // [units][T]
  int32_t* idx0;    // [units][B]
  int32_t* idx1;    // [units][B]
  float* rmean;     // [units][2][4 + 2D]   n_R, mean k, mean v of R0 / R
  float* m0;        // [units][4 + 2D + D*D] n0, mu_k0, mu_v0, C0
};

__host__ __device__ inline size_t rec_floats(int D) { return align_up(4 + 2 * (size_t)D + (size_t)D * D, 4); }

Layout make_layout(const mkv_geom& g, int T, int B, int W, int num_sms) {
  Layout L{};
  L.D = g.head_dim;
  L.G = g.group;
  L.W = W;
  L.RW = g.group * W;
  L.T = T;
  L.B = B;
  L.units = g.batch * g.n_kv_heads;
  long target = (2L * num_sms + L.units - 1) / L.units;
  long tiles = (T + kTT - 1) / kTT;
  if (target > tiles) target = tiles;
  if (target < 1) target = 1;
  L.chunk = static_cast<int>(((tiles + target - 1) / target) * kTT);
  L.n_chunks = (T + L.chunk - 1) / L.chunk;
  L.rec = rec_floats(L.D);
  return L;
}

size_t carve(Layout& L, void* ws) {
  uint8_t* base = static_cast<uint8_t*>(ws);
  size_t off = kHeaderBytes;
  auto take = [&](size_t bytes) {
    uint8_t* p = base ? base + off : nullptr;
    off += align_up(bytes, 256);
    return p;
  };
  const size_t U = L.units;
  L.rowpart = reinterpret_cast<float*>(take(U * L.n_chunks * L.RW * 2 * sizeof(float)));
  L.mpart = reinterpret_cast<float*>(take(U * L.n_chunks * L.rec * sizeof(float)));
  L.s = reinterpret_cast<float*>(take(U * (size_t)L.T * sizeof(float)));
  L.s2 = reinterpret_cast<float*>(take(U * (size_t)L.T * sizeof(float)));
  L.idx0 = reinterpret_cast<int32_t*>(take(U * (size_t)L.B * sizeof(int32_t)));
  L.idx1 = reinterpret_cast<int32_t*>(take(U * (size_t)L.B * sizeof(int32_t)));
  L.rmean = reinterpret_cast<float*>(take(U * 2 * (4 + 2 * (size_t)L.D) * sizeof(float)));
  L.m0 = reinterpret_cast<float*>(take(U * rec_floats(L.D) * sizeof(float)));
  return off;
}

// Is window row r = h*W + i allowed to see token t?
__device__ __forceinline__ bool visible(int t, int i, int T, int W, int causal) {
  return !causal || t <= T - W + i;
}

__device__ __forceinline__ bool is_protected(int t, int T, int W, int sink, int keep_window) {
  return t < sink || (keep_window && t >= T - W);
}

__host__ __device__ __forceinline__ int protected_count(int T, int W, int sink, int keep_window) {
  const int s = sink < T ? sink : T;
  const int w = keep_window ? (W < T ? W : T) : 0;
  const int overlap = s - (T - w) > 0 ? s - (T - w) : 0;
  return s + w - overlap;
}

// Load a [kTT][D] bf16 tile (rows t0..t0+rows-1) into fp32 shared memory with
// row stride D+1 (conflict-free both along rows and along columns).
template <int D>
__device__ __forceinline__ void load_tile(float* dst, const __nv_bfloat16* src, int rows, int tid, int nthr) {
  for (int idx = tid; idx < kTT * (D / 2); idx += nthr) {
    const int r = idx / (D / 2), c2 = (idx % (D / 2)) * 2;
    float2 f = make_float2(0.f, 0.f);
    if (r < rows) f = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(src + (size_t)r * D + c2));
    dst[r * (D + 1) + c2] = f.x;
    dst[r * (D + 1) + c2 + 1] = f.y;
  }
}

// Logits of 4 window rows (qT holds q*scale*log2e transposed, [D][RWpad]) for
// the 32 tokens of a tile, one token per lane.
template <int D>
__device__ __forceinline__ void logits4(float (&acc)[4], const float* qT, int RWp, int r0, const float* tK,
                                        int lane) {
#pragma unroll
  for (int i = 0; i < 4; ++i) acc[i] = 0.f;
#pragma unroll 8
  for (int c = 0; c < D; ++c) {
    const float kc = tK[lane * (D + 1) + c];
    const float4 q4 = *reinterpret_cast<const float4*>(qT + c * RWp + r0);
    acc[0] = fmaf(q4.x, kc, acc[0]);
    acc[1] = fmaf(q4.y, kc, acc[1]);
    acc[2] = fmaf(q4.z, kc, acc[2]);
    acc[3] = fmaf(q4.w, kc, acc[3]);
  }
}

// ----------------------------------------------------------------- stats
template <int D>
__global__ void __launch_bounds__(256) stats_kernel(const CompressArgs a, const Layout L) {
  constexpr int NT = 256;
  extern __shared__ __align__(16) float sm[];
  const int RWp = align_up(L.RW, 4);
  float* qT = sm;                          // [D][RWp]
  float* tK = qT + D * RWp;                // [32][D+1]
  float* tV = tK + kTT * (D + 1);          // [32][D+1]
  float* rowm = tV + kTT * (D + 1);        // [RWp]
  float* rowl = rowm + RWp;                // [RWp]
  const int chunk = blockIdx.x, u = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int t_begin = chunk * L.chunk;
  const int t_end = min(L.T, t_begin + L.chunk);
  const float qs = rsqrtf(static_cast<float>(D)) * kLog2e;

  const __nv_bfloat16* Qg = reinterpret_cast<const __nv_bfloat16*>(a.Q) + (size_t)u * L.RW * D;
  for (int idx = tid; idx < D * RWp; idx += NT) {
    const int c = idx / RWp, r = idx % RWp;
    qT[idx] = (r < L.RW) ? __bfloat162float(Qg[(size_t)r * D + c]) * qs : 0.f;
  }
  for (int r = tid; r < RWp; r += NT) {
    rowm[r] = -INFINITY;
    rowl[r] = 0.f;
  }
  // S accumulator: thread owns an (D/16) x 8 block: rows a0.., cols c0..
  constexpr int AR = D / 16;  // 8 at D=128, 4 at D=64
  const int a0 = (tid / 16) * AR, c0 = (tid % 16) * (D / 16);
  constexpr int CC = D / 16;
  float S[AR][CC];
#pragma unroll
  for (int i = 0; i < AR; ++i)
#pragma unroll
    for (int j = 0; j < CC; ++j) S[i][j] = 0.f;
  float colsum = 0.f;  // tid < D: sum k[:, tid]; D <= tid < 2D: sum v[:, tid-D]

  const __nv_bfloat16* Kg = reinterpret_cast<const __nv_bfloat16*>(a.K) + (size_t)u * L.T * D;
  const __nv_bfloat16* Vg = reinterpret_cast<const __nv_bfloat16*>(a.V) + (size_t)u * L.T * D;
  for (int t0 = t_begin; t0 < t_end; t0 += kTT) {
    const int rows = min(kTT, t_end - t0);
    __syncthreads();
    load_tile<D>(tK, Kg + (size_t)t0 * D, rows, tid, NT);
    load_tile<D>(tV, Vg + (size_t)t0 * D, rows, tid, NT);
    __syncthreads();
    // window-row statistics: each warp takes groups of 4 rows
    const int t = t0 + lane;
    for (int r0 = warp * 4; r0 < L.RW; r0 += 32) {
      float acc[4];
      logits4<D>(acc, qT, RWp, r0, tK, lane);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int r = r0 + i;
        if (r >= L.RW) break;
        const bool ok = lane < rows && visible(t, r % L.W, L.T, L.W, a.causal);
        const float x = ok ? acc[i] : -INFINITY;
        const float mt = warp_max(x);
        if (mt == -INFINITY) continue;
        const float mo = rowm[r];
        const float mn = fmaxf(mo, mt);
        const float p = ok ? fast_exp2(x - mn) : 0.f;
        const float ps = warp_sum(p);
        if (lane == 0) {
          rowl[r] = rowl[r] * fast_exp2(mo - mn) + ps;
          rowm[r] = mn;
        }
        __syncwarp();
      }
    }
    // moment sums
    for (int tt = 0; tt < rows; ++tt) {
      float va[AR], kc[CC];
#pragma unroll
      for (int i = 0; i < AR; ++i) va[i] = tV[tt * (D + 1) + a0 + i];
#pragma unroll
      for (int j = 0; j < CC; ++j) kc[j] = tK[tt * (D + 1) + c0 + j];
#pragma unroll
      for (int i = 0; i < AR; ++i)
#pragma unroll
        for (int j = 0; j < CC; ++j) S[i][j] = fmaf(va[i], kc[j], S[i][j]);
    }
    if (tid < D) {
      for (int tt = 0; tt < rows; ++tt) colsum += tK[tt * (D + 1) + tid];
    } else if (tid < 2 * D) {
      for (int tt = 0; tt < rows; ++tt) colsum += tV[tt * (D + 1) + tid - D];
    }
  }
  __syncthreads();
  float* rp = L.rowpart + ((size_t)u * L.n_chunks + chunk) * L.RW * 2;
  for (int r = tid; r < L.RW; r += NT) {
    rp[2 * r] = rowm[r];
    rp[2 * r + 1] = rowl[r];
  }
  // centred co-moment of this chunk
  float* rec = L.mpart + ((size_t)u * L.n_chunks + chunk) * L.rec;
  const float nc = static_cast<float>(t_end - t_begin);
  float* sums = tK;  // reuse: [0..D) sum k, [D..2D) sum v
  if (tid < 2 * D) sums[tid] = colsum;
  __syncthreads();
  if (tid == 0) rec[0] = nc;
  if (tid < D) {
    rec[4 + tid] = sums[tid] / nc;
    rec[4 + D + tid] = sums[D + tid] / nc;
  }
#pragma unroll
  for (int i = 0; i < AR; ++i)
#pragma unroll
    for (int j = 0; j < CC; ++j)
      rec[4 + 2 * D + (size_t)(a0 + i) * D + c0 + j] = S[i][j] - sums[D + a0 + i] * sums[c0 + j] / nc;
}

// ----------------------------------------------------------------- scores
template <int D>
__global__ void __launch_bounds__(256) scores_kernel(const CompressArgs a, const Layout L) {
  constexpr int NT = 256;
  extern __shared__ __align__(16) float sm[];
  const int RWp = align_up(L.RW, 4);
  float* qT = sm;                  // [D][RWp]
  float* tK = qT + D * RWp;        // [32][D+1]
  float* rowm = tK + kTT * (D + 1);
  float* rowil = rowm + RWp;       // 1 / l
  float* part = rowil + RWp;       // [8][32]
  const int chunk = blockIdx.x, u = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int t_begin = chunk * L.chunk;
  const int t_end = min(L.T, t_begin + L.chunk);
  const float qs = rsqrtf(static_cast<float>(D)) * kLog2e;
  const __nv_bfloat16* Qg = reinterpret_cast<const __nv_bfloat16*>(a.Q) + (size_t)u * L.RW * D;
  for (int idx = tid; idx < D * RWp; idx += NT) {
    const int c = idx / RWp, r = idx % RWp;
    qT[idx] = (r < L.RW) ? __bfloat162float(Qg[(size_t)r * D + c]) * qs : 0.f;
  }
  // merge the per-chunk row statistics
  const float* rp = L.rowpart + (size_t)u * L.n_chunks * L.RW * 2;
  for (int r = tid; r < RWp; r += NT) {
    float m = -INFINITY, l = 0.f;
    if (r < L.RW) {
      for (int c = 0; c < L.n_chunks; ++c) m = fmaxf(m, rp[((size_t)c * L.RW + r) * 2]);
      for (int c = 0; c < L.n_chunks; ++c) {
        const float mc = rp[((size_t)c * L.RW + r) * 2];
        if (mc != -INFINITY) l += rp[((size_t)c * L.RW + r) * 2 + 1] * fast_exp2(mc - m);
      }
    }
    rowm[r] = m;
    rowil[r] = (l > 0.f) ? 1.f / l : 0.f;
  }
  const __nv_bfloat16* Kg = reinterpret_cast<const __nv_bfloat16*>(a.K) + (size_t)u * L.T * D;
  float* s_out = L.s + (size_t)u * L.T;
  for (int t0 = t_begin; t0 < t_end; t0 += kTT) {
    const int rows = min(kTT, t_end - t0);
    __syncthreads();
    load_tile<D>(tK, Kg + (size_t)t0 * D, rows, tid, NT);
    __syncthreads();
    const int t = t0 + lane;
    float colp = 0.f;
    for (int r0 = warp * 4; r0 < L.RW; r0 += 32) {
      float acc[4];
      logits4<D>(acc, qT, RWp, r0, tK, lane);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int r = r0 + i;
        if (r < L.RW && lane < rows && visible(t, r % L.W, L.T, L.W, a.causal))
          colp += fast_exp2(acc[i] - rowm[r]) * rowil[r];
      }
    }
    part[warp * 32 + lane] = colp;
    __syncthreads();
    if (warp == 0) {
      float sum = 0.f;
#pragma unroll
      for (int w = 0; w < 8; ++w) sum += part[w * 32 + lane];
      // pool into aligned chunks of `pool` tokens (pool divides 32, tiles are aligned)
      for (int o = 1; o < a.pool; o <<= 1) sum += __shfl_xor_sync(kFull, sum, o);
      if (lane < rows) {
        s_out[t] = sum;
        if (a.diag_scores) a.diag_scores[(size_t)u * L.T + t] = sum;
      }
    }
  }
}

// ----------------------------------------------------------------- select
// One CTA (1024 threads) per unit: R = protected + the k highest keys among
// the other positions (ties to the lower position).  Writes R ascending to
// idx_out[u][0..B) and (n_R, mean k, mean v) of R to rmean_out.
constexpr int kSelThreads = 1024;

__device__ __forceinline__ int block_excl_scan(int flag, int* wsum, int* total) {
  // flag in {0,1}; returns exclusive prefix count in thread order
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const unsigned m = __ballot_sync(kFull, flag);
  const int in_warp = __popc(m & ((1u << lane) - 1u));
  if (lane == 0) wsum[warp] = __popc(m);
  __syncthreads();
  if (warp == 0) {
    const int v = wsum[lane];
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(kFull, x, o);
      if (lane >= o) x += y;
    }
    wsum[lane] = x - v;  // exclusive
    if (lane == 31) *total = x;
  }
  __syncthreads();
  const int r = wsum[warp] + in_warp;
  __syncthreads();
  return r;
}

template <int D>
__global__ void __launch_bounds__(kSelThreads) select_kernel(const CompressArgs a, const Layout L,
                                                             const float* scores, int32_t* idx_out,
                                                             float* rmean_out, int32_t* diag_idx) {
  __shared__ uint32_t hist[256];
  __shared__ int wsum[32];
  __shared__ int tot;
  __shared__ uint32_t s_prefix;
  __shared__ int s_need;
  const int u = blockIdx.x, tid = threadIdx.x;
  const int T = L.T, W = L.W;
  const float* sc = scores + (size_t)u * T;
  const int k = L.B - protected_count(T, W, a.sink, a.keep_window);  // >= 0 (validated), < candidates

  uint32_t prefix = 0, pmask = 0;
  int need = k;
  if (k > 0) {
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      for (int i = tid; i < 256; i += kSelThreads) hist[i] = 0;
      __syncthreads();
      for (int t = tid; t < T; t += kSelThreads) {
        if (is_protected(t, T, W, a.sink, a.keep_window)) continue;
        const uint32_t key = float_key(sc[t]);
        if ((key & pmask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (tid == 0) {
        int cum = 0, dg = 0;
        for (dg = 255; dg > 0; --dg) {
          if (cum + static_cast<int>(hist[dg]) >= need) break;
          cum += hist[dg];
        }
        s_need = need - cum;
        s_prefix = prefix | (static_cast<uint32_t>(dg) << shift);
      }
      __syncthreads();
      need = s_need;
      prefix = s_prefix;
      pmask |= 255u << shift;
      __syncthreads();
    }
  }
  // ascending output: selected = protected | key > K* | (key == K* and tie rank < need)
  int ties_before = 0, sel_before = 0;
  int32_t* out = idx_out + (size_t)u * L.B;
  for (int base = 0; base < T; base += kSelThreads) {
    const int t = base + tid;
    bool prot = false, tie = false, gt = false;
    if (t < T) {
      prot = is_protected(t, T, W, a.sink, a.keep_window);
      if (!prot && k > 0) {
        const uint32_t key = float_key(sc[t]);
        gt = key > prefix;
        tie = key == prefix;
      }
    }
    const int tr = block_excl_scan(tie ? 1 : 0, wsum, &tot);
    const int tie_total = tot;
    const bool sel = prot || gt || (tie && ties_before + tr < need);
    const int sr = block_excl_scan(sel ? 1 : 0, wsum, &tot);
    const int sel_total = tot;
    if (sel) {
      const int o = sel_before + sr;
      if (o < L.B) {
        out[o] = t;
        if (diag_idx) diag_idx[(size_t)u * L.B + o] = t;
      }
    }
    ties_before += tie_total;
    sel_before += sel_total;
  }
  __syncthreads();
  // mean key / value of R (thread c < D: key dim c; D <= thread < 2D: value dim)
  if (rmean_out) {
    float* rm = rmean_out + (size_t)u * (4 + 2 * D);
    const int nR = min(sel_before, L.B);
    if (tid < 2 * D) {
      const bool isv = tid >= D;
      const int c = isv ? tid - D : tid;
      const __nv_bfloat16* X = reinterpret_cast<const __nv_bfloat16*>(isv ? a.V : a.K) + (size_t)u * T * D;
      float acc = 0.f;
      for (int i = 0; i < nR; ++i) acc += __bfloat162float(X[(size_t)out[i] * D + c]);
      rm[4 + tid] = acc / static_cast<float>(nR);
    }
    if (tid == 0) rm[0] = static_cast<float>(nR);
  }
}

// ---------------------------------------------------------------- moments
// Moments of E = all \ R for 8 rows (value dims) of C per CTA.
template <int D>
__global__ void __launch_bounds__(256) moments_kernel(const CompressArgs a, const Layout L, const int32_t* idx,
                                                      const float* rmean, float* out_rec, mkv_moments out_mom,
                                                      int final_out) {
  constexpr int NT = 256, RB = 8;
  __shared__ float mk[D], mv[D], mkR[D], mvR[D];
  __shared__ float s_n;
  const int rb = blockIdx.x, u = blockIdx.y, tid = threadIdx.x;
  const float* recs = L.mpart + (size_t)u * L.n_chunks * L.rec;
  // totals over all tokens
  if (tid < 2 * D) {
    float num = 0.f, n = 0.f;
    for (int c = 0; c < L.n_chunks; ++c) {
      const float nc = recs[(size_t)c * L.rec];
      n += nc;
      num += nc * recs[(size_t)c * L.rec + 4 + tid];
    }
    if (tid < D) mk[tid] = num / n;
    else mv[tid - D] = num / n;
    if (tid == 0) s_n = n;
  }
  const float* rm = rmean + (size_t)u * (4 + 2 * D);
  if (tid < D) {
    mkR[tid] = rm[4 + tid];
    mvR[tid] = rm[4 + D + tid];
  }
  __syncthreads();
  const float n = s_n, nR = rm[0], nE = n - nR;
  const __nv_bfloat16* Kg = reinterpret_cast<const __nv_bfloat16*>(a.K) + (size_t)u * L.T * D;
  const __nv_bfloat16* Vg = reinterpret_cast<const __nv_bfloat16*>(a.V) + (size_t)u * L.T * D;
  const int32_t* ix = idx + (size_t)u * L.B;
  const int nRi = static_cast<int>(nR);
  for (int e = tid; e < RB * D; e += NT) {
    const int ar = rb * RB + e / D, c = e % D;
    // all-token co-moment: multi-way Chan merge of the chunk records
    float M = 0.f;
    for (int ch = 0; ch < L.n_chunks; ++ch) {
      const float* r = recs + (size_t)ch * L.rec;
      const float nc = r[0];
      M += r[4 + 2 * D + (size_t)ar * D + c] + nc * (r[4 + D + ar] - mv[ar]) * (r[4 + c] - mk[c]);
    }
    // retained-set co-moment
    float MR = 0.f;
    for (int i = 0; i < nRi; ++i) {
      const size_t row = (size_t)ix[i] * D;
      MR = fmaf(__bfloat162float(Vg[row + ar]) - mvR[ar], __bfloat162float(Kg[row + c]) - mkR[c], MR);
    }
    float CE = 0.f, mkE_c = 0.f, mvE_a = 0.f;
    if (nE > 0.f) {
      mkE_c = (n * mk[c] - nR * mkR[c]) / nE;
      mvE_a = (n * mv[ar] - nR * mvR[ar]) / nE;
      const float ME = M - MR - (nE * nR / n) * (mvR[ar] - mvE_a) * (mkR[c] - mkE_c);
      CE = ME / nE;
    }
    if (final_out) {
      out_mom.C[((size_t)u * D + ar) * D + c] = CE;
      if (c == 0) out_mom.mu_v[(size_t)u * D + ar] = (nE > 0.f) ? mvE_a : 0.f;
      if (rb == 0 && e < D) out_mom.mu_k[(size_t)u * D + c] = (nE > 0.f) ? mkE_c : 0.f;
    } else {
      float* o = out_rec + (size_t)u * rec_floats(D);
      o[4 + 2 * D + (size_t)ar * D + c] = CE;
      if (c == 0) o[4 + D + ar] = mvE_a;
      if (rb == 0 && e < D) o[4 + c] = mkE_c;
    }
  }
  if (rb == 0 && tid == 0) {
    if (final_out) out_mom.n[u] = static_cast<int32_t>(nE);
    else out_rec[(size_t)u * rec_floats(D)] = nE;
  }
}

// --------------------------------------------------------------- residual
template <int D>
__global__ void __launch_bounds__(256) residual_kernel(const CompressArgs a, const Layout L) {
  constexpr int NT = 256;
  extern __shared__ __align__(16) float sm[];
  float* Ct = sm;                   // [D][D] C0' transposed: Ct[c][a]
  float* tK = Ct + D * D;           // [32][D+1]
  float* part = tK + kTT * (D + 1); // [8][32]
  __shared__ float mv0[D];
  const int chunk = blockIdx.x, u = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int t_begin = chunk * L.chunk;
  const int t_end = min(L.T, t_begin + L.chunk);
  const float* m0 = L.m0 + (size_t)u * rec_floats(D);
  const float n0 = m0[0];
  const float tau = a.tau;
  for (int idx = tid; idx < D * D; idx += NT) {
    const int ar = idx / D, c = idx % D;
    float cv = (n0 > 0.f) ? m0[4 + 2 * D + idx] : 0.f;
    if (fabsf(cv * n0) < tau) cv = 0.f;
    Ct[c * D + ar] = cv;
  }
  if (tid < D) mv0[tid] = (n0 > 0.f) ? m0[4 + D + tid] : 0.f;
  const float scale = rsqrtf(static_cast<float>(D));
  const __nv_bfloat16* Kg = reinterpret_cast<const __nv_bfloat16*>(a.K) + (size_t)u * L.T * D;
  const __nv_bfloat16* Vg = reinterpret_cast<const __nv_bfloat16*>(a.V) + (size_t)u * L.T * D;
  const float* s = L.s + (size_t)u * L.T;
  float* s2 = L.s2 + (size_t)u * L.T;
  constexpr int AW = D / 8;  // output dims per warp
  for (int t0 = t_begin; t0 < t_end; t0 += kTT) {
    const int rows = min(kTT, t_end - t0);
    __syncthreads();
    load_tile<D>(tK, Kg + (size_t)t0 * D, rows, tid, NT);
    __syncthreads();
    float y[AW];
#pragma unroll
    for (int i = 0; i < AW; ++i) y[i] = 0.f;
    const int a0 = warp * AW;
#pragma unroll 4
    for (int c = 0; c < D; ++c) {
      const float kc = tK[lane * (D + 1) + c];
#pragma unroll
      for (int i = 0; i < AW; i += 4) {
        const float4 c4 = *reinterpret_cast<const float4*>(Ct + c * D + a0 + i);
        y[i] = fmaf(c4.x, kc, y[i]);
        y[i + 1] = fmaf(c4.y, kc, y[i + 1]);
        y[i + 2] = fmaf(c4.z, kc, y[i + 2]);
        y[i + 3] = fmaf(c4.w, kc, y[i + 3]);
      }
    }
    const int t = t0 + lane;
    float ss = 0.f;
    if (lane < rows) {
      const __nv_bfloat16* vrow = Vg + (size_t)t * D + a0;
#pragma unroll
      for (int i = 0; i < AW; ++i) {
        const float r = __bfloat162float(vrow[i]) - mv0[a0 + i] - scale * y[i];
        ss = fmaf(r, r, ss);
      }
    }
    part[warp * 32 + lane] = ss;
    __syncthreads();
    if (warp == 0 && lane < rows) {
      float tot = 0.f;
#pragma unroll
      for (int w = 0; w < 8; ++w) tot += part[w * 32 + lane];
      const float v = is_protected(t, L.T, L.W, a.sink, a.keep_window) ? 0.f : s[t] * sqrtf(tot);
      s2[t] = v;
      if (a.diag_score2) a.diag_score2[(size_t)u * L.T + t] = v;
    }
  }
}

// ----------------------------------------------------------------- gather
template <int D>
__global__ void __launch_bounds__(256) gather_kernel(const CompressArgs a, const Layout L, const int32_t* idx,
                                                     int count, int keep_all) {
  const int u = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = blockIdx.x * 8 + warp;
  if (i < count) {
    const int t = keep_all ? i : idx[(size_t)u * L.B + i];
    const __nv_bfloat16* Ks = reinterpret_cast<const __nv_bfloat16*>(a.K) + ((size_t)u * L.T + t) * D;
    const __nv_bfloat16* Vs = reinterpret_cast<const __nv_bfloat16*>(a.V) + ((size_t)u * L.T + t) * D;
    __nv_bfloat16* Kd = reinterpret_cast<__nv_bfloat16*>(a.cache.K) + ((size_t)u * a.cache.capacity + i) * D;
    __nv_bfloat16* Vd = reinterpret_cast<__nv_bfloat16*>(a.cache.V) + ((size_t)u * a.cache.capacity + i) * D;
    for (int c = lane * 2; c < D; c += 64) {
      *reinterpret_cast<__nv_bfloat162*>(Kd + c) = *reinterpret_cast<const __nv_bfloat162*>(Ks + c);
      *reinterpret_cast<__nv_bfloat162*>(Vd + c) = *reinterpret_cast<const __nv_bfloat162*>(Vs + c);
    }
    if (lane == 0) a.cache.pos[(size_t)u * a.cache.capacity + i] = t;
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) {
    a.cache.len[u] = count;
    a.cache.seen[u] = L.T;
  }
  if (keep_all && blockIdx.x == 0) {
    // nothing evicted: zero moments
    for (int e = threadIdx.x; e < D * D; e += blockDim.x) a.mom.C[(size_t)u * D * D + e] = 0.f;
    for (int e = threadIdx.x; e < D; e += blockDim.x) {
      a.mom.mu_k[(size_t)u * D + e] = 0.f;
      a.mom.mu_v[(size_t)u * D + e] = 0.f;
    }
    if (threadIdx.x == 0) a.mom.n[u] = 0;
  }
}

template <int D>
cudaError_t run(const CompressArgs& a, const mkv_geom& g, int num_sms, cudaStream_t st) {
  Layout L = make_layout(g, a.T, a.budget, a.window, num_sms);
  carve(L, a.ws);
  cudaError_t e;
  const dim3 cg(L.n_chunks, L.units);
  const int RWp = static_cast<int>(align_up(L.RW, 4));
  const bool keep_all = a.T <= a.budget;
  if (!keep_all || a.diag_scores != nullptr) {  // nothing to select when keep_all: score only if asked
    const size_t sm_stats = (size_t)(D * RWp + 2 * kTT * (D + 1) + 2 * RWp) * sizeof(float);
    e = cudaFuncSetAttribute(stats_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm_stats);
    if (e != cudaSuccess) return e;
    stats_kernel<D><<<cg, 256, sm_stats, st>>>(a, L);
    const size_t sm_scores = (size_t)(D * RWp + kTT * (D + 1) + 2 * RWp + 8 * 32) * sizeof(float);
    e = cudaFuncSetAttribute(scores_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm_scores);
    if (e != cudaSuccess) return e;
    scores_kernel<D><<<cg, 256, sm_scores, st>>>(a, L);
  }
  if (keep_all) {
    gather_kernel<D><<<dim3((a.T + 7) / 8, L.units), 256, 0, st>>>(a, L, nullptr, a.T, 1);
    return cudaGetLastError();
  }
  select_kernel<D><<<L.units, kSelThreads, 0, st>>>(a, L, L.s, L.idx0, L.rmean, a.diag_idx1);
  const int32_t* final_idx = L.idx0;
  const float* final_rmean = L.rmean;
  if (a.mi) {
    moments_kernel<D><<<dim3(D / 8, L.units), 256, 0, st>>>(a, L, L.idx0, L.rmean, L.m0, a.mom, 0);
    const size_t sm_res = (size_t)(D * D + kTT * (D + 1) + 8 * 32) * sizeof(float);
    e = cudaFuncSetAttribute(residual_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sm_res);
    if (e != cudaSuccess) return e;
    residual_kernel<D><<<cg, 256, sm_res, st>>>(a, L);
    float* rm1 = L.rmean + (size_t)L.units * (4 + 2 * D);
    select_kernel<D><<<L.units, kSelThreads, 0, st>>>(a, L, L.s2, L.idx1, rm1, nullptr);
    final_idx = L.idx1;
    final_rmean = rm1;
  }
  moments_kernel<D><<<dim3(D / 8, L.units), 256, 0, st>>>(a, L, final_idx, final_rmean, nullptr, a.mom, 1);
  gather_kernel<D><<<dim3((a.budget + 7) / 8, L.units), 256, 0, st>>>(a, L, final_idx, a.budget, 0);
  return cudaGetLastError();
}

}  // namespace

size_t compress_workspace_bytes(const mkv_geom& g, int32_t T, const mkv_compress_params& p, int num_sms) {
  Layout L = make_layout(g, T, p.budget, p.window, num_sms);
  return carve(L, nullptr);
}

cudaError_t launch_compress(const CompressArgs& a, const mkv_geom& g, size_t ws_bytes, int num_sms,
                            cudaStream_t stream) {
  (void)ws_bytes;
  if (g.head_dim == 128) return run<128>(a, g, num_sms, stream);
  if (g.head_dim == 64) return run<64>(a, g, num_sms, stream);
  return cudaErrorInvalidValue;
}

}  // namespace mkv
