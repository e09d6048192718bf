// Decode step, ticket form: retained-cache attention merged with the moment
// correction (Algorithm 1 Phase 2; Eqs. jensen, fhat, fused; log-domain merge
// of App. C.2).  mkv_decode_step runs this kernel only when the split CTAs of
// a unit cannot form a thread-block cluster (or a test forces it); the
// cluster kernel in decode_cl.cu is the normal path.
//
// Grid (S, h_kv, b): every CTA serves all G query heads of one KV head
// (GQA grouping, so K/V rows are read once per unit) over one contiguous
// split of the retained rows.  Rows stream from HBM through a 3-stage ring of
// 64-row tiles, each filled by 2-D TMA tensor copies (boxes of 64 rows x 64
// columns, 128-byte swizzle, mbarrier completion); the swizzle makes every
// shared-memory fragment load below bank-conflict-free.  Each warp takes 16
// rows of a tile: S = Q K^T and O += P V run on the tensor cores
// (mma.m16n8k16, bf16 in, fp32 accumulate) with the G query heads as the M
// rows; P is split into bf16 hi + lo parts so the mixing weights keep ~16
// bits.  The moment term S_tilde q / (n sqrt d) is spread over the same CTAs:
// CTA s computes rows [s*D/S, ...) of C'q for all G heads on the tensor cores
// (C' rows split into bf16 hi + lo parts as the A operand, the q fragments as
// B), so C (64 KB fp32 at d=128, or its bf16 copy in the C16 variant) is read
// once per unit, concurrently with the K/V stream.  The appended token is
// attended to by the last split, which also writes its row.  The last CTA of
// a unit to finish (atomic ticket, no waiting) merges the S partial (m, l, o)
// records with the moment pseudo-partial (log n + scale q.mu_k, f_hat_E) by
// log-sum-exp, writes the output and updates the length.
//
// Launched as a programmatic dependent of the previous kernel in the stream:
// barrier set-up overlaps its tail, and every global read waits on
// griddepcontrol.wait (the previous grid complete, its writes visible).
#include <algorithm>

#include "common.cuh"
#include "kernels.h"
#include "warp_mma.cuh"

namespace mkv {

namespace {

constexpr int kThreads = 128;  // 4 warps x 16 rows of each 64-row tile
constexpr int kStages = 3;
constexpr int kTT = kDecodeTile;
constexpr unsigned kFull = 0xffffffffu;

// A rows 8..15 are zero (at most 8 query heads per KV head): registers a1, a3 = 0
__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a2, uint32_t b0, uint32_t b1) {
  mma_m16n8k16(d, a0, 0u, a2, 0u, b0, b1);
}

// (hi, lo) bf16 pair parts of two floats: hi = bf16(x), lo = bf16(x - hi)
__device__ __forceinline__ void split_bf16x2(float x, float y, uint32_t& hi, uint32_t& lo) {
  hi = pack_bf16x2(x, y);
  lo = pack_bf16x2(bf16_residual(x), bf16_residual(y));
}

// Per-warp online-softmax state for head g = lane/4 (meaningful when g < G):
// running max m (log2 domain), sum l, and O[g][nt*8 + 2t + {0,1}] in o[nt][0..1].
template <int D>
struct WarpState {
  float m, l;
  float o[D / 8][4];
};

// 16 rows [row0, row0 + 16) of a shared-memory tile; rows >= `rows` are masked.
template <int D, int G>
__device__ __forceinline__ void process16(WarpState<D>& st, const uint32_t (&qa)[D / 16][2],
                                          const uint8_t* tK, const uint8_t* tV, int row0, int rows,
                                          float qscale, int lane) {
  const int g = lane >> 2, t = lane & 3;
  float s[2][4];
#pragma unroll
  for (int nt = 0; nt < 2; ++nt) {
    s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
    const int r = row0 + nt * 8 + g;
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      const uint32_t b0 = *reinterpret_cast<const uint32_t*>(tK + swz_off(r, kk * 16 + 2 * t, kTT));
      const uint32_t b1 = *reinterpret_cast<const uint32_t*>(tK + swz_off(r, kk * 16 + 8 + 2 * t, kTT));
      mma_bf16(s[nt], qa[kk][0], qa[kk][1], b0, b1);
    }
  }
  float x[4];
#pragma unroll
  for (int nt = 0; nt < 2; ++nt)
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int tok = row0 + nt * 8 + 2 * t + j;
      x[nt * 2 + j] = (tok < rows) ? s[nt][j] * qscale : -INFINITY;
    }
  float tmax = fmaxf(fmaxf(x[0], x[1]), fmaxf(x[2], x[3]));
  tmax = fmaxf(tmax, __shfl_xor_sync(kFull, tmax, 1));
  tmax = fmaxf(tmax, __shfl_xor_sync(kFull, tmax, 2));
  const float mnew = fmaxf(st.m, tmax);
  const float alpha = (mnew == -INFINITY) ? 1.f : fast_exp2(st.m - mnew);
  float p[4], ps = 0.f;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    p[i] = (x[i] == -INFINITY) ? 0.f : fast_exp2(x[i] - mnew);
    ps += p[i];
  }
  ps += __shfl_xor_sync(kFull, ps, 1);
  ps += __shfl_xor_sync(kFull, ps, 2);
  st.l = st.l * alpha + ps;
  st.m = mnew;
#pragma unroll
  for (int nt = 0; nt < D / 8; ++nt) {
    st.o[nt][0] *= alpha;
    st.o[nt][1] *= alpha;
  }
  // P as bf16 hi + lo (A operand: tokens 2t, 2t+1 and 8+2t, 8+2t+1 of row g)
  const uint32_t ph0 = pack_bf16x2(p[0], p[1]), ph2 = pack_bf16x2(p[2], p[3]);
  const float r0 = p[0] - __bfloat162float(__float2bfloat16_rn(p[0]));
  const float r1 = p[1] - __bfloat162float(__float2bfloat16_rn(p[1]));
  const float r2 = p[2] - __bfloat162float(__float2bfloat16_rn(p[2]));
  const float r3 = p[3] - __bfloat162float(__float2bfloat16_rn(p[3]));
  const uint32_t pl0 = pack_bf16x2(r0, r1), pl2 = pack_bf16x2(r2, r3);
  const int mi = lane >> 3, mr = lane & 7;
  const int vr = row0 + (mi & 1) * 8 + mr;
#pragma unroll
  for (int np = 0; np < D / 16; ++np) {
    uint32_t vb[4];
    ldsm_x4_t(vb, tV + swz_off(vr, np * 16 + (mi >> 1) * 8, kTT));
    mma_bf16(st.o[2 * np], ph0, ph2, vb[0], vb[1]);
    mma_bf16(st.o[2 * np], pl0, pl2, vb[0], vb[1]);
    mma_bf16(st.o[2 * np + 1], ph0, ph2, vb[2], vb[3]);
    mma_bf16(st.o[2 * np + 1], pl0, pl2, vb[2], vb[3]);
  }
}

template <int D, int G, bool C16, bool EARLY>
__global__ void __launch_bounds__(kThreads) decode_kernel(const DecodeArgs a, const __grid_constant__ CUtensorMap tmK,
                                                          const __grid_constant__ CUtensorMap tmV) {
  constexpr int PS = D + 4;  // partial record: o[D], m (log2 domain), l
  constexpr int kTileBytes = kTT * D * 2;
  extern __shared__ __align__(128) uint8_t dsmem_raw[];
  // the 128-byte swizzle pattern repeats every 1024 bytes: align the ring to it
  uint8_t* dsmem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dsmem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sK = dsmem;                          // [stage][box][kTT][128 B]
  uint8_t* sV = dsmem + kStages * kTileBytes;
  __shared__ float sFp[2][4][16][8];  // C'q partial sums: [m16 tile][warp][row][head]
  __shared__ float sSbar[G];
  __shared__ float sM[G], sL[G];
  __shared__ __align__(8) uint64_t bars[kStages];
  __shared__ int sTicket;

  const int s = blockIdx.x, kv = blockIdx.y, b = blockIdx.z;
  const int u = b * a.n_kv + kv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const float scale = rsqrtf(static_cast<float>(D));

  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) mbar_init(&bars[i], 1);
    mbar_fence_init();
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
  }
  if (tid == 0 && !EARLY) {
    // Before the dependency wait: this split's retained rows and moment rows
    // were written by earlier calls, not by the kernel this launch waits on
    // (that one produces this step's query and token), so its first tiles
    // (at most 2 kStages: more would only crowd L2 when many units stream at
    // once) are pulled into L2 now, while that kernel still runs.  A prefetch
    // is only a hint and L2 is the point of coherence: a length read that
    // races with a writer only moves the prefetched range; the loads after
    // the wait read the current values.
    int lp = __ldcg(a.len + u);
    lp = lp < 0 ? 0 : (lp > a.cap ? a.cap : lp);
    const int tp = (lp + kTT - 1) / kTT;
    const int per = (tp + a.S - 1) / a.S;
    const int pb = min(lp, s * per * kTT), pe = min(lp, pb + min(per, 2 * kStages) * kTT);
    if (pe > pb) {
      const size_t off = ((size_t)u * a.cap + pb) * D * 2;
      const uint32_t bytes = static_cast<uint32_t>((pe - pb) * D * 2);
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(static_cast<const uint8_t*>(a.K) + off),
                   "r"(bytes) : "memory");
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(static_cast<const uint8_t*>(a.V) + off),
                   "r"(bytes) : "memory");
    }
    if (a.correction && a.n != nullptr && a.order == 1) {
      const int rp = (D + a.S - 1) / a.S, c0 = s * rp, c1 = min(D, c0 + rp);
      if (c1 > c0) {
        const void* base = C16 ? static_cast<const void*>(a.C16 + ((size_t)u * D + c0) * D)
                               : static_cast<const void*>(a.C + ((size_t)u * D + c0) * D);
        asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(base),
                     "r"((uint32_t)((c1 - c0) * D * (C16 ? 2 : 4))) : "memory");
      }
    }
  }
  // ---- the unit's cache length, its first tiles and its moment rows.  With
  // EARLY the caller guarantees that the kernels that may still run when
  // this launch starts (in a layer chain: the previous layer's) write
  // neither this cache nor these moments, so they are read, and the first
  // tile copies go out, before the dependency wait, overlapping that
  // kernel's tail; only the query and the new token, which it may produce,
  // wait.  Otherwise everything is read after the wait.
  const bool corr = a.correction != 0 && a.n != nullptr;
  // Moment rows [r0, r1) of this split: C'q on the tensor cores.  The rows
  // form m16 tiles (A = C' rows, split into bf16 hi + lo parts: about 16
  // significant bits); B is q itself, whose fragments are the qa registers
  // (column n = head).  Up to two tiles (many splits, small batches): warp w
  // takes the k-steps [w*KPW, (w+1)*KPW) of each tile, its fragments are
  // loaded now, and the four partial sums meet in shared memory.  More tiles
  // (few splits, large batches): warp w takes whole tiles w, w + 4, ....
  constexpr int KPW = D / 64;
  const int rpc = (D + a.S - 1) / a.S;
  const int r0 = s * rpc, r1 = min(D, r0 + rpc);
  const int n_mt = (r1 - r0 + 15) / 16;
  const bool do_c = corr && a.order == 1;
  const bool split_k = n_mt <= 2;
  // C[row][c0], C[row][c0 + 1] as float2, from C or from its bf16 copy; with
  // the operand form of C' (cs), the bits of its (hi, lo) words
  constexpr bool c16 = C16;  // moment rows read from the bf16 copy of C
  const bool cs = !c16 && a.Cs != nullptr;
  auto ld_c2 = [&](int row, int c0) -> float2 {
    const size_t off = ((size_t)u * D + row) * D + c0;
    if constexpr (c16) return __bfloat1622float2(__ldg(reinterpret_cast<const __nv_bfloat162*>(a.C16 + off)));
    else if (cs) return __ldg(reinterpret_cast<const float2*>(a.Cs + off / 2));
    else return __ldg(reinterpret_cast<const float2*>(a.C + off));
  };
  float2 cfr[2][KPW][4];
  // mu_v of the (row, head) pairs this thread finishes in the two-tile case
  constexpr int kPairs = 2 * 16 * 8 / kThreads;  // at most 32 rows x 8 heads
  float muv_pre[kPairs];
  // mu_k at this lane's q dims (warp 1 computes scale q . mu_k for its head)
  float2 mkp[D / 16][2];
  int n_e = 0;
  auto load_moments = [&]() {
    const int g = lane >> 2, t = lane & 3;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int ra = r0 + j * 16 + g, rb = ra + 8;
#pragma unroll
      for (int kp = 0; kp < KPW; ++kp) {
        const int c0 = (warp * KPW + kp) * 16 + 2 * t;
        const bool va = do_c && split_k && ra < r1, vb = do_c && split_k && rb < r1;
        cfr[j][kp][0] = va ? ld_c2(ra, c0) : make_float2(0.f, 0.f);
        cfr[j][kp][1] = vb ? ld_c2(rb, c0) : make_float2(0.f, 0.f);
        cfr[j][kp][2] = va ? ld_c2(ra, c0 + 8) : make_float2(0.f, 0.f);
        cfr[j][kp][3] = vb ? ld_c2(rb, c0 + 8) : make_float2(0.f, 0.f);
      }
    }
    if (do_c && !split_k && tid == 0 && r1 > r0) {  // whole-tile case: the rows are read after the tiles
      const void* base = c16  ? static_cast<const void*>(a.C16 + ((size_t)u * D + r0) * D)
                         : cs ? static_cast<const void*>(a.Cs + ((size_t)u * D + r0) * D / 2)
                              : static_cast<const void*>(a.C + ((size_t)u * D + r0) * D);
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(base),
                   "r"((uint32_t)((r1 - r0) * D * (c16 ? 2 : 4)))
                   : "memory");
    }
#pragma unroll
    for (int j = 0; j < kPairs; ++j) {
      const int idx = tid + j * kThreads, row = r0 + idx / G;
      muv_pre[j] = (do_c && split_k && row < r1) ? __ldg(a.mu_v + (size_t)u * D + row) : 0.f;
    }
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      const bool v = corr && warp == 1 && g < G;
      mkp[kk][0] = v ? __ldg(reinterpret_cast<const float2*>(a.mu_k + (size_t)u * D + kk * 16 + 2 * t))
                     : make_float2(0.f, 0.f);
      mkp[kk][1] = v ? __ldg(reinterpret_cast<const float2*>(a.mu_k + (size_t)u * D + kk * 16 + 8 + 2 * t))
                     : make_float2(0.f, 0.f);
    }
    n_e = corr ? __ldcg(a.n + u) : 0;
  };
  // the cached rows are split into whole tiles over the S CTAs; one thread
  // fills a stage: a 64-row box per 64 columns, for K and for V (rows past
  // the unit's slab belong to the next unit or are zero-filled by the TMA
  // unit; they are masked below)
  int len_read = 0, len0 = 0, t_begin = 0, n_cached = 0, n_tiles = 0, row_base = 0;
  auto issue = [&](int it) {
    const int st = it % kStages;
    mbar_arrive_expect_tx(&bars[st], 2u * kTileBytes);
#pragma unroll
    for (int bx = 0; bx < D / 64; ++bx) {
      tma_load_2d(sK + st * kTileBytes + bx * kTT * 128, &tmK, bx * 64, row_base + it * kTT, &bars[st]);
      tma_load_2d(sV + st * kTileBytes + bx * kTT * 128, &tmV, bx * 64, row_base + it * kTT, &bars[st]);
    }
  };
  auto load_len_and_issue = [&]() {
    len_read = __ldcg(a.len + u);
    len0 = len_read;
    if (len0 < 0 || len0 > a.cap) {  // corrupt cache state: never read past the slab
      if (tid == 0 && s == 0) record_error(a.ws, MKV_ERR_CAPACITY, u);
      len0 = len0 < 0 ? 0 : a.cap;
    }
    const int tiles_total = (len0 + kTT - 1) / kTT;
    const int tiles_per = (tiles_total + a.S - 1) / a.S;
    t_begin = min(len0, s * tiles_per * kTT);
    n_cached = min(len0, t_begin + tiles_per * kTT) - t_begin;
    n_tiles = (n_cached + kTT - 1) / kTT;
    row_base = u * a.cap + t_begin;
    if (tid == 0)
      for (int i = 0; i < min(kStages, n_tiles); ++i) issue(i);
  };
  if constexpr (EARLY) {
    load_len_and_issue();
    if (tid == 0) {  // the split's next tiles past the first stages (up to 2 kStages): into L2 now
      const int first = min(kStages, n_tiles);
      if (min(n_tiles, 2 * kStages) > first) {
        const size_t off = ((size_t)row_base + first * kTT) * D * 2;
        const uint32_t bytes = static_cast<uint32_t>((min(n_cached, 2 * kStages * kTT) - first * kTT) * D * 2);
        asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(static_cast<const uint8_t*>(a.K) + off),
                     "r"(bytes) : "memory");
        asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(static_cast<const uint8_t*>(a.V) + off),
                     "r"(bytes) : "memory");
      }
    }
    load_moments();
  }
  grid_dependency_wait();
  grid_launch_dependents();

  // ---- the query: the A operand, rows = heads (g = lane/4 < G), 16 dims per k-step
  const __nv_bfloat16* qg = reinterpret_cast<const __nv_bfloat16*>(a.q) + ((size_t)u * G) * D;
  uint32_t qa[D / 16][2];
  {
    const int g = lane >> 2, t = lane & 3;
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      qa[kk][0] = (g < G) ? *reinterpret_cast<const uint32_t*>(qg + g * D + kk * 16 + 2 * t) : 0u;
      qa[kk][1] = (g < G) ? *reinterpret_cast<const uint32_t*>(qg + g * D + kk * 16 + 8 + 2 * t) : 0u;
    }
  }
  if constexpr (!EARLY) {
    load_moments();
    load_len_and_issue();
  } else if (tid == 0 && s == 0 && __ldcg(a.len + u) != len_read) {
    record_error(a.ws, MKV_ERR_INVALID_ARG, u);  // the cache changed under an early load
  }
  const bool has_new = a.k_new != nullptr;
  const bool use_m = n_e > 0;
  // the appended token is attended to by the last CTA (which holds the
  // fewest rows), whose threads fetch it now: threads 0..D/8-1 hold 16 bytes
  // of k each, the next D/8 threads 16 bytes of v
  const bool own_new = has_new && s == a.S - 1;
  uint4 new_part = make_uint4(0u, 0u, 0u, 0u);
  if (own_new && tid < D / 4) {
    const __nv_bfloat16* src = reinterpret_cast<const __nv_bfloat16*>(tid < D / 8 ? a.k_new : a.v_new) + (size_t)u * D;
    new_part = reinterpret_cast<const uint4*>(src)[tid % (D / 8)];
  }
  if (use_m && warp == 1) {  // scale * q . mu_k per head from the qa fragments (lanes 4h..4h+3)
    const int g = lane >> 2;
    float acc = 0.f;
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      const __nv_bfloat162 q0 = *reinterpret_cast<const __nv_bfloat162*>(&qa[kk][0]);
      const __nv_bfloat162 q1 = *reinterpret_cast<const __nv_bfloat162*>(&qa[kk][1]);
      acc = fmaf(__low2float(q0), mkp[kk][0].x, fmaf(__high2float(q0), mkp[kk][0].y, acc));
      acc = fmaf(__low2float(q1), mkp[kk][1].x, fmaf(__high2float(q1), mkp[kk][1].y, acc));
    }
    acc += __shfl_xor_sync(kFull, acc, 1);
    acc += __shfl_xor_sync(kFull, acc, 2);
    if ((lane & 3) == 0 && g < G) sSbar[g] = acc * scale;
  }
  const float tau = a.tau;
  const float nf = static_cast<float>(n_e);
  // one m16 x n8 product over the k-steps [kk0, kk0 + nk) from fragments in
  // registers (clamp of Eq. fused's C' applied here)
  auto mma_c = [&](float (&d)[4], const float2 (&f)[4], int kk) {
    uint32_t hi[4], lo[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      if (cs) {  // already clamped and split
        hi[i] = __float_as_uint(f[i].x);
        lo[i] = __float_as_uint(f[i].y);
      } else {
        const float x = (fabsf(f[i].x * nf) < tau) ? 0.f : f[i].x;
        const float y = (fabsf(f[i].y * nf) < tau) ? 0.f : f[i].y;
        split_bf16x2(x, y, hi[i], lo[i]);
      }
    }
    // the q fragment of k-step kk, selected without indexing the register
    // array by a runtime value (which would move qa to local memory)
    uint32_t b0 = 0u, b1 = 0u;
#pragma unroll
    for (int k = 0; k < D / 16; ++k) {
      b0 = (k == kk) ? qa[k][0] : b0;
      b1 = (k == kk) ? qa[k][1] : b1;
    }
    mma_m16n8k16(d, hi[0], hi[1], hi[2], hi[3], b0, b1);
    mma_m16n8k16(d, lo[0], lo[1], lo[2], lo[3], b0, b1);  // zero for a bf16 copy of C
  };
  if (use_m && do_c && split_k) {
    const int g = lane >> 2, t = lane & 3;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      if (j < n_mt) {  // warp-uniform; no early exit, so cfr stays in registers
        float d[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int kp = 0; kp < KPW; ++kp) mma_c(d, cfr[j][kp], warp * KPW + kp);
        float(*fp)[8] = sFp[j][warp];
        fp[g][2 * t] = d[0];
        fp[g][2 * t + 1] = d[1];
        fp[g + 8][2 * t] = d[2];
        fp[g + 8][2 * t + 1] = d[3];
      }
    }
  }
  __syncthreads();
  // f_hat_E[h][row] = mu_v[row] + scale * (C'q_h)[row]
  if (use_m && do_c) {
    float* fdst = a.fhat + (size_t)u * G * D;
    if (split_k) {
      const int n_pairs = (r1 - r0) * G;
#pragma unroll
      for (int j = 0; j < kPairs; ++j) {
        const int idx = tid + j * kThreads;
        if (idx < n_pairs) {
          const int rr = idx / G, h = idx % G;
          const float* fp = &sFp[rr >> 4][0][rr & 15][h];
          const float cq = fp[0] + fp[16 * 8] + fp[2 * 16 * 8] + fp[3 * 16 * 8];
          fdst[h * D + r0 + rr] = muv_pre[j] + scale * cq;
        }
      }
    } else {
      const int g = lane >> 2, t = lane & 3;
      for (int mt = warp; mt < n_mt; mt += 4) {
        const int ra = r0 + mt * 16 + g, rb = ra + 8;
        const bool va = ra < r1, vb = rb < r1;
        float2 f[D / 16][4];
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const int c0 = kk * 16 + 2 * t;
          f[kk][0] = va ? ld_c2(ra, c0) : make_float2(0.f, 0.f);
          f[kk][1] = vb ? ld_c2(rb, c0) : make_float2(0.f, 0.f);
          f[kk][2] = va ? ld_c2(ra, c0 + 8) : make_float2(0.f, 0.f);
          f[kk][3] = vb ? ld_c2(rb, c0 + 8) : make_float2(0.f, 0.f);
        }
        const float mva = va ? __ldg(a.mu_v + (size_t)u * D + ra) : 0.f;
        const float mvb = vb ? __ldg(a.mu_v + (size_t)u * D + rb) : 0.f;
        float d[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) mma_c(d, f[kk], kk);
        // lane holds rows (g, g + 8) x heads (2t, 2t + 1)
        if (2 * t < G) {
          if (va) fdst[(2 * t) * D + ra] = mva + scale * d[0];
          if (vb) fdst[(2 * t) * D + rb] = mvb + scale * d[2];
        }
        if (2 * t + 1 < G) {
          if (va) fdst[(2 * t + 1) * D + ra] = mva + scale * d[1];
          if (vb) fdst[(2 * t + 1) * D + rb] = mvb + scale * d[3];
        }
      }
    }
  }

  // ---- retained rows
  WarpState<D> st;
  st.m = -INFINITY;
  st.l = 0.f;
#pragma unroll
  for (int nt = 0; nt < D / 8; ++nt) st.o[nt][0] = st.o[nt][1] = st.o[nt][2] = st.o[nt][3] = 0.f;
  const float qscale = scale * kLog2e;
  bool ok = true;
  int it = 0;
  for (; it < n_tiles; ++it) {
    const int stg = it % kStages;
    const int rows = min(kTT, n_cached - it * kTT);
    const bool got = mbar_wait(&bars[stg], (it / kStages) & 1, a.polls);
    if (!__syncthreads_and(got)) {
      ok = false;
      break;
    }
    if (rows < kTT) {  // ragged tile: zero the unused V rows (P is 0 there, V must be finite)
      for (int i = tid; i < (kTT - rows) * (D / 8); i += kThreads) {
        const int r = rows + i / (D / 8), c = (i % (D / 8)) * 8;  // whole rows: layout-free
        *reinterpret_cast<uint4*>(sV + stg * kTileBytes + (c >> 6) * kTT * 128 + r * 128 + (c & 63) * 2) =
            make_uint4(0u, 0u, 0u, 0u);
      }
      __syncthreads();
    }
    process16<D, G>(st, qa, sK + stg * kTileBytes, sV + stg * kTileBytes, warp * 16, rows, qscale, lane);
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
    st.m = -INFINITY;
    st.l = 0.f;
#pragma unroll
    for (int nt = 0; nt < D / 8; ++nt) st.o[nt][0] = st.o[nt][1] = 0.f;
  }
  if (own_new) {  // the appended token: row 0 of stage 0 (free now), rows 1..15 zero
    // a row is one 128-byte line per 64-column box; the swizzle permutes the
    // 16-byte chunks within a row, so zero rows are zero in any order
    for (int i = tid; i < 16 * (D / 8); i += kThreads) {
      const int r = i / (D / 8), c = (i % (D / 8)) * 8;
      const uint32_t off = (c >> 6) * kTT * 128 + r * 128 + (((c & 63) >> 3) << 4);
      *reinterpret_cast<uint4*>(sK + off) = make_uint4(0u, 0u, 0u, 0u);
      *reinterpret_cast<uint4*>(sV + off) = make_uint4(0u, 0u, 0u, 0u);
    }
    __syncthreads();
    if (tid < D / 4) {
      const int c = (tid % (D / 8)) * 8;
      *reinterpret_cast<uint4*>((tid < D / 8 ? sK : sV) + swz_off(0, c, kTT)) = new_part;
    }
    __syncthreads();
    if (warp == 0) process16<D, G>(st, qa, sK, sV, 0, 1, qscale, lane);
    if (len0 + 1 <= a.cap && tid < D / 4) {  // nobody reads this cache row during the step
      __nv_bfloat16* dst =
          reinterpret_cast<__nv_bfloat16*>(tid < D / 8 ? a.K : a.V) + ((size_t)u * a.cap + len0) * D;
      reinterpret_cast<uint4*>(dst)[tid % (D / 8)] = new_part;
    }
  }

  // ---- merge the 4 warps into this CTA's partial record (through the free tile ring)
  float* sRed = reinterpret_cast<float*>(dsmem);  // [4][G][D + 2]
  __syncthreads();
  {
    const int g = lane >> 2, t = lane & 3;
    if (g < G) {
      float* rw = sRed + (warp * G + g) * (D + 2);
#pragma unroll
      for (int nt = 0; nt < D / 8; ++nt) {
        rw[nt * 8 + 2 * t] = st.o[nt][0];
        rw[nt * 8 + 2 * t + 1] = st.o[nt][1];
      }
      if (t == 0) {
        rw[D] = st.m;
        rw[D + 1] = st.l;
      }
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

  const size_t rec_floats = (size_t)a.S * G * PS;
  bool staged = false;
  const float* src = nullptr;
  float* sF = nullptr;  // [G][D] f_hat_E rows (or mu_v for order 0)
  float* sP = reinterpret_cast<float*>(dsmem);
  {
    // ---- ticket: the last CTA of this unit merges everything
    __threadfence();
    __syncthreads();
    if (tid == 0) sTicket = static_cast<int>(atomicAdd(&a.counters[u], 1u));
    __syncthreads();
    if (sTicket != a.S - 1) return;
    __threadfence();
    if (tid == 0) a.counters[u] = 0u;

    // combine the S partial records: stage them in shared memory with one
    // round of loads when they fit in the (free) tile ring, else read them
    // in place
    const float* pu = a.partial + (size_t)u * a.S * G * PS;
    staged = rec_floats * 4 + (2 * a.S * G + G * D) * 4 <= (size_t)kStages * 2 * kTileBytes;
    src = pu;
    sF = sP;
    if (staged) {
      sF = sP + rec_floats;
      for (size_t i = tid; i < rec_floats / 4; i += kThreads)
        reinterpret_cast<float4*>(sP)[i] = __ldcg(reinterpret_cast<const float4*>(pu) + i);
      if (use_m) {
        for (int i = tid; i < G * D / 4; i += kThreads)
          reinterpret_cast<float4*>(sF)[i] =
              (a.order == 1) ? __ldcg(reinterpret_cast<const float4*>(a.fhat + (size_t)u * G * D) + i)
                             : __ldg(reinterpret_cast<const float4*>(a.mu_v + (size_t)u * D) + (i % (D / 4)));
      }
      src = sP;
    }
  }
  float* sW = staged ? sF + G * D : sP;  // [S][G] max, then weight
  float* sLs = sW + a.S * G;             // [S][G] sums
  __syncthreads();
  for (int i = tid; i < a.S * G; i += kThreads) {
    sW[i] = staged ? src[(size_t)i * PS + D] : __ldcg(src + (size_t)i * PS + D);
    sLs[i] = staged ? src[(size_t)i * PS + D + 1] : __ldcg(src + (size_t)i * PS + D + 1);
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
    float fh[4];
    if (use_m) {
#pragma unroll
      for (int k = 0; k < 4; ++k)
        fh[k] = staged ? sF[h * D + d0 + k]
                       : ((a.order == 1) ? __ldcg(a.fhat + ((size_t)u * G + h) * D + d0 + k)
                                         : a.mu_v[(size_t)u * D + d0 + k]);
    }
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
    for (int sp = 0; sp < a.S; ++sp) {
      const float w = sW[sp * G + h];
      const float* rec = src + ((size_t)sp * G + h) * PS + d0;
      const float4 o = staged ? *reinterpret_cast<const float4*>(rec) : __ldcg(reinterpret_cast<const float4*>(rec));
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

  if (has_new && tid == 0) {  // the row itself was written by the CTA that attended to it
    if (len0 + 1 > a.cap) {
      record_error(a.ws, MKV_ERR_CAPACITY, u);
    } else {
      a.pos[(size_t)u * a.cap + len0] = a.seen[u];
      a.seen[u] = a.seen[u] + 1;
      a.len[u] = len0 + 1;
    }
  }
}

template <int D, int G, bool C16, bool EARLY>
cudaError_t launch_dgc(const DecodeArgs& args, cudaStream_t stream) {
  DecodeArgs a = args;
  a.polls = pipeline_poll_limit();
  const size_t ring = (size_t)2 * kStages * kTT * D * 2 + 1024;  // + alignment slack
  cudaError_t e = cudaFuncSetAttribute(decode_kernel<D, G, C16, EARLY>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(ring));
  if (e != cudaSuccess) return e;
  // the cache slabs of all units as one [units * cap][D] matrix
  const uint64_t rows = (uint64_t)a.batch * a.n_kv * a.cap;
  CUtensorMap tmK, tmV;
  if (!encode_tmap_bf16(&tmK, a.K, D, rows, (uint64_t)D * 2, 64, kTT) ||
      !encode_tmap_bf16(&tmV, a.V, D, rows, (uint64_t)D * 2, 64, kTT))
    return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(a.S, a.n_kv, a.batch);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = ring;
  cfg.stream = stream;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, decode_kernel<D, G, C16, EARLY>, a, tmK, tmV);
}

template <int D, int G>
cudaError_t launch_dg(const DecodeArgs& a, cudaStream_t stream) {
  if (a.early)
    return a.C16 != nullptr ? launch_dgc<D, G, true, true>(a, stream) : launch_dgc<D, G, false, true>(a, stream);
  return a.C16 != nullptr ? launch_dgc<D, G, true, false>(a, stream) : launch_dgc<D, G, false, false>(a, stream);
}

}  // namespace

namespace {
__global__ void __launch_bounds__(256) pack_bf16_kernel(const float* __restrict__ C, __nv_bfloat16* __restrict__ C16,
                                                        size_t n4) {
  for (size_t i = (size_t)blockIdx.x * 256 + threadIdx.x; i < n4; i += (size_t)gridDim.x * 256) {
    const float4 v = reinterpret_cast<const float4*>(C)[i];
    __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y), hi = __floats2bfloat162_rn(v.z, v.w);
    uint2 w;
    w.x = *reinterpret_cast<uint32_t*>(&lo);
    w.y = *reinterpret_cast<uint32_t*>(&hi);
    reinterpret_cast<uint2*>(C16)[i] = w;
  }
}
// The operand form of C' (Eq. fused with the App. C.2 clamp): per column
// pair, the (hi, lo) bf16x2 words the decode kernels feed to the tensor cores,
// computed exactly as they compute them from C at a step (split_bf16x2 of the
// clamped pair).  Grid-stride over float4s of C: two pairs each.
__global__ void __launch_bounds__(256) pack_split_kernel(const float* __restrict__ C, const int32_t* __restrict__ n,
                                                         float tau, uint2* __restrict__ Cs, size_t n4, int per_unit4) {
  for (size_t i = (size_t)blockIdx.x * 256 + threadIdx.x; i < n4; i += (size_t)gridDim.x * 256) {
    const float nf = static_cast<float>(n[i / per_unit4]);
    const float4 v = reinterpret_cast<const float4*>(C)[i];
    const float c[4] = {v.x, v.y, v.z, v.w};
    uint32_t hi[2], lo[2];
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const float x = (fabsf(c[2 * j] * nf) < tau) ? 0.f : c[2 * j];
      const float y = (fabsf(c[2 * j + 1] * nf) < tau) ? 0.f : c[2 * j + 1];
      split_bf16x2(x, y, hi[j], lo[j]);
    }
    reinterpret_cast<uint4*>(Cs)[i] = make_uint4(hi[0], lo[0], hi[1], lo[1]);
  }
}
}  // namespace

cudaError_t launch_pack_split(const float* C, const int32_t* n, float tau, uint2* Cs, int units, int D,
                              cudaStream_t stream) {
  const int per_unit4 = D * D / 4;
  const size_t n4 = (size_t)units * per_unit4;
  const int blocks = static_cast<int>(std::min<size_t>((n4 + 255) / 256, 65535));
  if (n4 > 0) pack_split_kernel<<<blocks, 256, 0, stream>>>(C, n, tau, Cs, n4, per_unit4);
  return cudaGetLastError();
}

cudaError_t launch_pack_bf16(const float* C, __nv_bfloat16* C16, size_t n, cudaStream_t stream) {
  const size_t n4 = n / 4;  // d * d is a multiple of 4
  const int blocks = static_cast<int>(std::min<size_t>((n4 + 255) / 256, 65535));
  if (n4 > 0) pack_bf16_kernel<<<blocks, 256, 0, stream>>>(C, C16, n4);
  return cudaGetLastError();
}

// Split count of the ticket kernel: up to two CTAs per SM, one tile per CTA
// up to ten tiles, at least two tiles per CTA beyond, and at most 12 splits,
// past which the merge costs more than the extra parallelism saves.
int decode_splits(const mkv_geom& g, int32_t capacity, int num_sms) {
  const long units = (long)g.batch * g.n_kv_heads;
  const long tiles = ((long)capacity + 1 + kTT - 1) / kTT;
  const long by_tiles = tiles <= 10 ? tiles : std::max(10L, (tiles + 1) / 2);
  long S = std::min<long>(std::min(by_tiles, 12L), 2L * num_sms / units);
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
  a.S_cl = decode_cluster_splits(g, capacity, num_sms, a.early);
}

cudaError_t launch_decode(const DecodeArgs& a, int head_dim, int group, cudaStream_t stream) {
  if (a.S_cl > 0 && g_force_ticket_merge.load() == 0) return launch_decode_cluster(a, head_dim, group, stream);
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
