// Decode step, cluster form: retained-cache attention merged with the moment
// correction (Algorithm 1 Phase 2; Eqs. jensen, fhat, fused; log-domain
// merge of App. C.2).  This is the kernel every mkv_decode_step runs when
// the S split CTAs of a unit can form one thread-block cluster (S <= 8); the
// ticket kernel in decode.cu covers the rest.
//
// Grid (S, h_kv, b), cluster (S, 1, 1), five warps per CTA.  CTA s of a unit
// takes a contiguous run of 64-row tiles of the unit's retained rows and all
// G query heads of its KV head (GQA grouping: each K/V row is read once per
// unit).
//
// - Warp 4 (producer) fills a ring of 2-3 stages with 2-D TMA copies
//   (64-row x 64-column boxes, 128-byte swizzle) under full/empty mbarrier
//   pairs, so the attending warps never meet at a block barrier.
// - Warps 0-3 each take 16 rows of every tile.  Both products run on the
//   tensor cores with the keys and the value dims as the 16-row side and the
//   G heads as the 8-column side: S^T = K q^T (K through ldmatrix, q in
//   registers), then O^T += V^T P^T (V through transposed ldmatrix, P^T moved
//   into operand layout by movmatrix, split into bf16 hi + lo parts so the
//   mixing weights keep about 16 bits).  A lane's accumulators then belong
//   to heads 2t and 2t + 1, the same heads whose softmax state it keeps.
// - Merge: CTA r owns output dims [r*D/S, (r+1)*D/S) in 16-dim blocks, and
//   also the rows of C' with those indices, so its part of the moment term
//   f_hat_E = mu_v + scale C' q is computed where it is used.  The four
//   warps' states first merge within the CTA (through the ring, free by
//   then); the CTA's unnormalised state (m, l per head, O) then goes to the
//   owners as 16-byte asynchronous stores into their shared memory, counted
//   by an mbarrier in each owner, and each owner merges its dims with one
//   output per thread: the S CTA states, the appended token as one more state
//   (m = its score, l = 1, O = v_new), and the moment pseudo-state (log n +
//   scale q.mu_k, f_hat_E).  (Scalar stores through generic pointers into
//   another CTA's shared memory measured several microseconds for the same
//   data.)
//
// Launched as a programmatic dependent of the previous kernel in the stream.
// With mkv_decode_params.early_load the cache length, the first tiles and
// the moment rows are read before the dependency wait; the query and the new
// token always after it.  Every mbarrier wait is bounded: running out
// records MKV_ERR_TIMEOUT, and the CTA still sends its (empty) state to the
// owners and drains its copies in flight before it exits.
#include <algorithm>
#include <mutex>

#include "common.cuh"
#include "kernels.h"
#include "warp_mma.cuh"

namespace mkv {

namespace {

constexpr int kConsumerWarps = 4;               // warps 0-3 attend over the tiles
constexpr int kLoaderWarp = kConsumerWarps;      // warp 4: tile copies, new token, per-head weights
                                                 // (warp 5 shares the C'q blocks with it)
constexpr int kClThreads = (kConsumerWarps + 2) * 32;
constexpr int kRows = kDecodeTile;  // rows per stage
constexpr int kMaxStages = 3;
constexpr int kMaxSplits = 8;  // a portable cluster
constexpr float kNegInf = -INFINITY;
constexpr float kSlack = 8.f;  // log2 headroom of the softmax reference (weights <= 2^8)

// Output dims owned by CTA r of S: 16-dim blocks [r*MT/S, (r+1)*MT/S), MT = D/16.
__host__ __device__ __forceinline__ int own_lo(int r, int S, int MT) { return r * MT / S; }

// log2 and reciprocal on the special-function unit (relative error ~2^-22)
__device__ __forceinline__ float fast_log2(float x) {
  float y;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
__device__ __forceinline__ float fast_rcp(float x) {
  float y;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// The most dims any CTA owns.
__host__ __device__ constexpr int cl_own_dims(int D, int S) { return 16 * ((D / 16 + S - 1) / S); }
__host__ __device__ constexpr size_t cl_stage_bytes(int D) { return (size_t)2 * kRows * D * 2; }
// Shared memory beyond the ring: receive areas, f_hat_E rows, mu_v and v_new of the owned dims.
__host__ __device__ constexpr size_t cl_extra_bytes(int D, int G, int S) {
  return (size_t)S * G * cl_own_dims(D, S) * 4 + (size_t)S * G * 2 * 4 + (size_t)cl_own_dims(D, S) * G * 4 +
         (size_t)2 * cl_own_dims(D, S) * 4;
}
// Three stages when two CTAs (of this launch and the next one in a layer
// chain) still fit on an SM, else two.
constexpr size_t kClSmemTarget = 112 * 1024;
__host__ __device__ constexpr int cl_stages(int D, int G, int S) {
  return 3 * cl_stage_bytes(D) + cl_extra_bytes(D, G, S) + 1024 <= kClSmemTarget ? 3 : 2;
}
__host__ __device__ constexpr size_t cl_smem_bytes(int D, int G, int S) {
  return cl_stages(D, G, S) * cl_stage_bytes(D) + cl_extra_bytes(D, G, S) + 1024;  // + alignment slack
}

template <int D, int G, bool C16, bool EARLY, bool CS>
__global__ void __launch_bounds__(kClThreads, 2)
    decode_cl_kernel(const DecodeArgs a, const __grid_constant__ CUtensorMap tmK,
                     const __grid_constant__ CUtensorMap tmV) {
  constexpr int MT = D / 16;  // 16-dim blocks of the output (and 16-row blocks of C')
  constexpr int KS = D / 16;  // k-steps of a dot product over the head dim
  constexpr int kTileBytes = kRows * D * 2;
  const int S = a.S;
  const int NST = cl_stages(D, G, S);
  const int OD = cl_own_dims(D, S);
  extern __shared__ __align__(128) uint8_t dsm_raw[];
  // the 128-byte swizzle pattern repeats every 1024 bytes: align the ring to it
  uint8_t* ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dsm_raw) + 1023) & ~uintptr_t(1023));
  float* rcv_o = reinterpret_cast<float*>(ring + (size_t)NST * 2 * kTileBytes);  // [S][G][OD] CTA states
  float* rcv_ml = rcv_o + (size_t)S * G * OD;                                    // [S][G][2] (m, l)
  float* sF = rcv_ml + (size_t)S * G * 2;                                        // [OD][G] f_hat_E
  float* sVn = sF + (size_t)OD * G;                                              // [OD] v_new
  float* sMuv = sVn + OD;                                                        // [OD] mu_v
  __shared__ __align__(8) uint64_t full[kMaxStages], empty[kMaxStages], recv;
  __shared__ float sE[G], sSn[G];   // log2 of the moment weight n exp(scale q.mu_k); new token's logit
  __shared__ float sMuk[D], sKn[D];
  __shared__ int sOwner[MT], sLo[MT], sFail;

  const int s = blockIdx.x, kv = blockIdx.y, b = blockIdx.z;
  const int u = b * a.n_kv + kv;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, t = lane & 3;
  const bool producer = warp == kLoaderWarp;
  const bool side = warp >= kLoaderWarp;  // the loader and moment warps
  const float scale = rsqrtf(static_cast<float>(D));
  const int mlo = own_lo(s, S, MT), mhi = own_lo(s + 1, S, MT);
  const int nmt = mhi - mlo, own_d = nmt * 16;

  if (tid == 0) {
    for (int i = 0; i < NST; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kConsumerWarps);
    }
    // the receive barrier completes when every CTA's state for the owned dims has landed
    mbar_init(&recv, 1);
    mbar_arrive_expect_tx(&recv, own_d > 0 ? static_cast<uint32_t>(S * G * (own_d + 2) * 4) : 0u);
    mbar_fence_init();
    sFail = 0;
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
  }
  if (tid < MT) {  // owner of each 16-dim block and that owner's first block
    int r = 0;
    while (r + 1 < S && own_lo(r + 1, S, MT) <= tid) ++r;
    sOwner[tid] = r;
    sLo[tid] = own_lo(r, S, MT);
  }
  __syncthreads();
  cluster_arrive_relaxed();  // paired with the wait before the first remote store

  const bool corr = a.correction != 0 && a.n != nullptr;
  const bool do_c = corr && a.order == 1;
  const bool has_new = a.k_new != nullptr;
  // Moments and cache lengths are read again at every step while the cache
  // rows stream through: the former stay in L2 (evict_last), the latter give
  // way first (evict_first).
  const uint64_t pol_keep = l2_evict_last(), pol_stream = l2_evict_first();

  // ---- state read before (EARLY) or after the dependency wait
  int len_read = 0, len0 = 0, n_tiles = 0, n_cached = 0, row_base = 0, seen0 = 0, n_e = 0, issued = 0;
  float2 cf[KS][4];  // side warps: C' fragments of one owned 16-row block, all k-steps
  // with the operand form of C' (mkv_moments_pack_split; the CS variant) a
  // fragment's float2 holds the bits of its (hi, lo) words, already clamped
  // and split
  static_assert(!(C16 && CS), "one form of C");
  constexpr bool cs = CS;
  auto load_cf = [&](int j) {
    const int ra = (mlo + j) * 16 + g, rb = ra + 8;
    const bool va = do_c && j < nmt;
#pragma unroll
    for (int kk = 0; kk < KS; ++kk) {
      const int c0 = kk * 16 + 2 * t;
      auto ld = [&](int row, int col) -> float2 {
        const size_t off = ((size_t)u * D + row) * D + col;
        if constexpr (C16) {
          const uint32_t w = ldg_hint(reinterpret_cast<const uint32_t*>(a.C16 + off), pol_keep);
          return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w));
        } else if constexpr (CS) {
          return ldg_hint(reinterpret_cast<const float2*>(a.Cs + off / 2), pol_keep);
        } else {
          return ldg_hint(reinterpret_cast<const float2*>(a.C + off), pol_keep);
        }
      };
      cf[kk][0] = va ? ld(ra, c0) : make_float2(0.f, 0.f);
      cf[kk][1] = va ? ld(rb, c0) : make_float2(0.f, 0.f);
      cf[kk][2] = va ? ld(ra, c0 + 8) : make_float2(0.f, 0.f);
      cf[kk][3] = va ? ld(rb, c0 + 8) : make_float2(0.f, 0.f);
    }
  };
  auto issue = [&](int i) {  // producer lane 0: tile i of the split into stage i % NST
    const int st = i % NST;
    uint8_t* dk = ring + (size_t)st * 2 * kTileBytes;
    mbar_arrive_expect_tx(&full[st], 2u * kTileBytes);
#pragma unroll
    for (int bx = 0; bx < D / 64; ++bx) {
      tma_load_2d_hint(dk + bx * kRows * 128, &tmK, bx * 64, row_base + i * kRows, &full[st], pol_stream);
      tma_load_2d_hint(dk + kTileBytes + bx * kRows * 128, &tmV, bx * 64, row_base + i * kRows, &full[st], pol_stream);
    }
  };
  auto prologue = [&]() {
    len_read = ldcg_hint(a.len + u, pol_keep);
    len0 = len_read;
    if (len0 < 0 || len0 > a.cap) {  // corrupt cache state: never read past the slab
      if (tid == 0 && s == 0) record_error(a.ws, MKV_ERR_CAPACITY, u);
      len0 = len0 < 0 ? 0 : a.cap;
    }
    const int tiles = (len0 + kRows - 1) / kRows, per = (tiles + S - 1) / S;
    const int tb = min(tiles, s * per), te = min(tiles, tb + per);
    n_tiles = te - tb;
    n_cached = max(0, min(len0, te * kRows) - tb * kRows);
    row_base = u * a.cap + tb * kRows;
    n_e = corr ? ldcg_hint(a.n + u, pol_keep) : 0;
    if (!side) return;
    if (producer) {
      if (lane == 0) {
        for (; issued < min(NST, n_tiles); ++issued) issue(issued);
        // the split's next tiles into L2 now (at most NST more: a longer run
        // would only crowd L2 when many units stream at once)
        const int pe = min(n_tiles, 2 * NST);
        if (pe > issued) {
          const size_t off = ((size_t)row_base + issued * kRows) * D * 2;
          const uint32_t bytes = static_cast<uint32_t>((min(n_cached, pe * kRows) - issued * kRows) * D * 2);
          asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(static_cast<const uint8_t*>(a.K) + off),
                       "r"(bytes) : "memory");
          asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(static_cast<const uint8_t*>(a.V) + off),
                       "r"(bytes) : "memory");
        }
        if (do_c && nmt > 2) {  // C' rows past the first two blocks are read later: into L2 now
          const void* base = C16  ? static_cast<const void*>(a.C16 + ((size_t)u * D + (mlo + 2) * 16) * D)
                             : cs ? static_cast<const void*>(a.Cs + ((size_t)u * D + (mlo + 2) * 16) * D / 2)
                                  : static_cast<const void*>(a.C + ((size_t)u * D + (mlo + 2) * 16) * D);
          asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(base),
                       "r"((uint32_t)((nmt - 2) * 16 * D * (C16 ? 2 : 4))) : "memory");
        }
        if (s == 0 && has_new) seen0 = ldcg_hint(a.seen + u, pol_keep);
      }
      if constexpr (EARLY) {
        // The query and the new token may be written by the kernel this
        // launch waits on, so they are read after the wait; their lines are
        // only pulled into L2 now.  A prefetch is a hint and L2 is the point
        // of coherence: a line the earlier kernel writes afterwards is
        // updated in L2, and the loads after the wait see its final value.
        constexpr int kQLines = G * D * 2 / 128, kNLines = D * 2 / 128;
        const char* line = nullptr;
        if (lane < kQLines) line = static_cast<const char*>(a.q) + (size_t)u * G * D * 2 + lane * 128;
        else if (has_new && lane < kQLines + 2 * kNLines) {
          const int j = lane - kQLines;
          line = static_cast<const char*>(j < kNLines ? a.k_new : a.v_new) + (size_t)u * D * 2 + (j % kNLines) * 128;
        }
        if (line != nullptr) asm volatile("prefetch.global.L2 [%0];" ::"l"(line));
      }
    }
    if (corr) {
      // this warp's first C' block (blocks alternate between the loader and
      // moment warps), issued without waiting for the count n (unused when
      // n = 0); the moment warp also stages the owned mu_v rows and mu_k (its
      // stores wait for those loads, the loader must not: its tile copies
      // and refills come first)
      load_cf(warp - kLoaderWarp);
      if (!producer) {
        for (int i = lane; i < own_d; i += 32) sMuv[i] = ldg_hint(a.mu_v + (size_t)u * D + mlo * 16 + i, pol_keep);
        for (int i = lane; i < D; i += 32) sMuk[i] = ldg_hint(a.mu_k + (size_t)u * D + i, pol_keep);
      }
    }
  };
  if constexpr (EARLY) prologue();
  grid_dependency_wait();
  // The next kernel in the stream may be scheduled from here on (in a layer
  // chain its CTAs then load their tiles while this launch runs).  Not
  // earlier: a launch that starts before this one's predecessor has finished
  // could read a cache that predecessor is still appending to.
  grid_launch_dependents();
  if constexpr (!EARLY) prologue();

  // ---- the query as the B operand of both products: column g = head, 16 dims per k-step
  const __nv_bfloat16* qg = reinterpret_cast<const __nv_bfloat16*>(a.q) + (size_t)u * G * D;
  uint32_t qa[KS][2];
#pragma unroll
  for (int kk = 0; kk < KS; ++kk) {
    qa[kk][0] = (g < G) ? *reinterpret_cast<const uint32_t*>(qg + g * D + kk * 16 + 2 * t) : 0u;
    qa[kk][1] = (g < G) ? *reinterpret_cast<const uint32_t*>(qg + g * D + kk * 16 + 8 + 2 * t) : 0u;
  }
  const bool use_m = n_e > 0;
  const float qscale = scale * kLog2e;

  if (side) {
    // the new token: 16 bytes of k (lanes < D/8) or v (lanes < D/4) per lane
    uint4 kvc = make_uint4(0u, 0u, 0u, 0u);
    if (producer && has_new && lane < D / 4)
      kvc = reinterpret_cast<const uint4*>(
          reinterpret_cast<const __nv_bfloat16*>(lane < D / 8 ? a.k_new : a.v_new) + (size_t)u * D)[lane % (D / 8)];
    if (producer) {
      // refills: stage i % NST is free once the four attending warps released tile i - NST
      if (lane == 0) {
        for (; issued < n_tiles; ++issued) {
          if (!mbar_wait(&empty[issued % NST], ((issued / NST) - 1) & 1, a.polls)) {
            sFail = 1;
            break;
          }
          issue(issued);
        }
      }
      __syncwarp();
    }
    __syncwarp();
    named_sync(3, 64);  // the moment warp's mu_v and mu_k rows are in place
    if (use_m) {
      // f_hat_E rows of the owned blocks, blocks alternating between the two
      // side warps: mu_v + scale C'q on the tensor cores (A = C' rows split
      // into bf16 hi + lo parts, clamp of Eq. fused applied here, or both
      // read ready-made from the operand form; B = the q fragments), written
      // as sF[row][head].  Four independent accumulator
      // chains (k-step parity x part): these products share the tensor pipe
      // with an attending warp's tiles.
      const float nf = static_cast<float>(n_e), tau = a.tau;
      for (int j = warp - kLoaderWarp; j < nmt; j += 2) {
        if (j > 1) load_cf(j);
        float dc[4][4] = {};
        if constexpr (CS) {
          if (do_c) {  // operand words as loaded
#pragma unroll
            for (int kk = 0; kk < KS; ++kk) {
              mma_m16n8k16(dc[kk & 1], __float_as_uint(cf[kk][0].x), __float_as_uint(cf[kk][1].x),
                           __float_as_uint(cf[kk][2].x), __float_as_uint(cf[kk][3].x), qa[kk][0], qa[kk][1]);
              mma_m16n8k16(dc[2 + (kk & 1)], __float_as_uint(cf[kk][0].y), __float_as_uint(cf[kk][1].y),
                           __float_as_uint(cf[kk][2].y), __float_as_uint(cf[kk][3].y), qa[kk][0], qa[kk][1]);
            }
          }
        } else if (do_c) {
#pragma unroll
          for (int kk = 0; kk < KS; ++kk) {
            uint32_t hi[4], lo[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const float x = (fabsf(cf[kk][i].x * nf) < tau) ? 0.f : cf[kk][i].x;
              const float y = (fabsf(cf[kk][i].y * nf) < tau) ? 0.f : cf[kk][i].y;
              hi[i] = pack_bf16x2(x, y);
              lo[i] = pack_bf16x2(bf16_residual(x), bf16_residual(y));
            }
            mma_m16n8k16(dc[kk & 1], hi[0], hi[1], hi[2], hi[3], qa[kk][0], qa[kk][1]);
            if constexpr (!C16) mma_m16n8k16(dc[2 + (kk & 1)], lo[0], lo[1], lo[2], lo[3], qa[kk][0], qa[kk][1]);
          }
        }
        float d[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) d[i] = (dc[0][i] + dc[1][i]) + (dc[2][i] + dc[3][i]);
        const int ra = j * 16 + g, rb = ra + 8;  // local rows (owned dims)
        const float mva = sMuv[ra], mvb = sMuv[rb];
        if (2 * t < G) {
          sF[ra * G + 2 * t] = fmaf(scale, d[0], mva);
          sF[rb * G + 2 * t] = fmaf(scale, d[2], mvb);
        }
        if (2 * t + 1 < G) {
          sF[ra * G + 2 * t + 1] = fmaf(scale, d[1], mva);
          sF[rb * G + 2 * t + 1] = fmaf(scale, d[3], mvb);
        }
      }
    }
    if (producer) {
      if (has_new && lane < D / 4) {  // the token as floats: all of k, the owned dims of v
        const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&kvc);
        const int c0 = (lane % (D / 8)) * 8;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float2 f = __bfloat1622float2(h2[i]);
          if (lane < D / 8) {
            sKn[c0 + 2 * i] = f.x;
            sKn[c0 + 2 * i + 1] = f.y;
          } else if (c0 >= mlo * 16 && c0 < mlo * 16 + own_d) {
            sVn[c0 - mlo * 16 + 2 * i] = f.x;
            sVn[c0 - mlo * 16 + 2 * i + 1] = f.y;
          }
        }
        // the appended row itself (nobody reads cache row len0 during this step)
        if (s == S - 1 && len0 + 1 <= a.cap)
          reinterpret_cast<uint4*>(reinterpret_cast<__nv_bfloat16*>(lane < D / 8 ? a.K : a.V) +
                                   ((size_t)u * a.cap + len0) * D)[lane % (D / 8)] = kvc;
      }
      __syncwarp();
      // per head: log2 of the moment weight n exp(scale q.mu_k) and the new
      // token's logit (log2 domain), from this lane's q dims
      float dm2[2] = {0.f, 0.f}, dn2[2] = {0.f, 0.f};
#pragma unroll
      for (int kk = 0; kk < KS; ++kk) {
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
          const __nv_bfloat162 q2 = *reinterpret_cast<const __nv_bfloat162*>(&qa[kk][hf]);
          const int c = kk * 16 + hf * 8 + 2 * t;
          if (use_m) dm2[hf] = fmaf(__low2float(q2), sMuk[c], fmaf(__high2float(q2), sMuk[c + 1], dm2[hf]));
          if (has_new) dn2[hf] = fmaf(__low2float(q2), sKn[c], fmaf(__high2float(q2), sKn[c + 1], dn2[hf]));
        }
      }
      float dm = dm2[0] + dm2[1], dn = dn2[0] + dn2[1];
      dm += __shfl_xor_sync(0xffffffffu, dm, 1);
      dm += __shfl_xor_sync(0xffffffffu, dm, 2);
      dn += __shfl_xor_sync(0xffffffffu, dn, 1);
      dn += __shfl_xor_sync(0xffffffffu, dn, 2);
      if (t == 0 && g < G) {
        sE[g] = use_m ? fast_log2(static_cast<float>(n_e)) + dm * qscale : kNegInf;
        sSn[g] = has_new ? dn * qscale : kNegInf;
      }
    }
    if (!producer && EARLY && s == 0 && lane == 0 && ldcg_hint(a.len + u, pol_keep) != len_read)
      record_error(a.ws, MKV_ERR_INVALID_ARG, u);  // the cache changed under an early load
    cluster_wait_acquire();
  } else {
    // ---- attending warps: rows [warp*16, warp*16 + 16) of every tile
    const int r0 = warp * 16;
    float m0 = kNegInf, m1 = kNegInf, l0 = 0.f, l1 = 0.f;  // heads 2t, 2t + 1 (log2 domain)
    float o[MT][4];  // O^T: dims (mt*16 + g, + 8) x heads (2t, 2t + 1)
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
    bool ok = true;
    for (int it = 0; it < n_tiles; ++it) {
      const int st = it % NST;
      const bool got = mbar_wait(&full[st], (it / NST) & 1, a.polls);
      if (!__all_sync(0xffffffffu, got)) {
        ok = false;
        break;
      }
      const int rows = min(kRows, n_cached - it * kRows);
      const uint8_t* tK = ring + (size_t)st * 2 * kTileBytes;
      uint8_t* tV = ring + (size_t)st * 2 * kTileBytes + kTileBytes;
      if (rows > r0) {
        if (rows < r0 + 16) {  // ragged last tile: zero this warp's V rows past the end (P is 0 there)
          for (int i = lane; i < (r0 + 16 - rows) * (D / 8); i += 32) {
            const int r = rows + i / (D / 8), c = (i % (D / 8)) * 8;  // whole rows: layout-free
            *reinterpret_cast<uint4*>(tV + (c >> 6) * kRows * 128 + r * 128 + (c & 63) * 2) =
                make_uint4(0u, 0u, 0u, 0u);
          }
          __syncwarp();
        }
        // S^T = K q^T over 16 keys: four accumulator chains (k-step mod 4)
        float c0[4] = {0.f, 0.f, 0.f, 0.f}, c1[4] = {0.f, 0.f, 0.f, 0.f};
        float c2[4] = {0.f, 0.f, 0.f, 0.f}, c3[4] = {0.f, 0.f, 0.f, 0.f};
        const int kr = r0 + (lane & 7) + ((lane >> 3) & 1) * 8, kc = (lane >> 4) * 8;
#pragma unroll
        for (int kk = 0; kk < KS; ++kk) {
          uint32_t k4[4];
          ldsm_x4(k4, tK + swz_off(kr, kk * 16 + kc, kRows));
          if ((kk & 3) == 0) mma_m16n8k16(c0, k4[0], k4[1], k4[2], k4[3], qa[kk][0], qa[kk][1]);
          else if ((kk & 3) == 1) mma_m16n8k16(c1, k4[0], k4[1], k4[2], k4[3], qa[kk][0], qa[kk][1]);
          else if ((kk & 3) == 2) mma_m16n8k16(c2, k4[0], k4[1], k4[2], k4[3], qa[kk][0], qa[kk][1]);
          else mma_m16n8k16(c3, k4[0], k4[1], k4[2], k4[3], qa[kk][0], qa[kk][1]);
        }
        // lane (g, t): keys r0 + g (x0, x1) and r0 + g + 8 (x2, x3), heads 2t (x0, x2) and 2t + 1 (x1, x3)
        const bool va = r0 + g < rows, vb = r0 + g + 8 < rows;
        const float x0 = va ? ((c0[0] + c2[0]) + (c1[0] + c3[0])) * qscale : kNegInf;
        const float x1 = va ? ((c0[1] + c2[1]) + (c1[1] + c3[1])) * qscale : kNegInf;
        const float x2 = vb ? ((c0[2] + c2[2]) + (c1[2] + c3[2])) * qscale : kNegInf;
        const float x3 = vb ? ((c0[3] + c2[3]) + (c1[3] + c3[3])) * qscale : kNegInf;
        // The softmax reference m of a head only has to be common to the
        // head's keys; any value gives the same normalised result.  It moves
        // (with the rescaling of O and l) only when a score exceeds it by more
        // than kSlack in log2 units, so the weights stay at most 2^kSlack and
        // most tiles skip the cross-lane maximum.
        const float lm0 = fmaxf(x0, x2), lm1 = fmaxf(x1, x3);
        if (__any_sync(0xffffffffu, lm0 > m0 + kSlack || lm1 > m1 + kSlack)) {
          float mx0 = lm0, mx1 = lm1;
#pragma unroll
          for (int off = 4; off < 32; off <<= 1) {
            mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, off));
            mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, off));
          }
          const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
          const float al0 = (mn0 == kNegInf) ? 1.f : fast_exp2(m0 - mn0);
          const float al1 = (mn1 == kNegInf) ? 1.f : fast_exp2(m1 - mn1);
          l0 *= al0;
          l1 *= al1;
          m0 = mn0;
          m1 = mn1;
#pragma unroll
          for (int mt = 0; mt < MT; ++mt) {
            o[mt][0] *= al0;
            o[mt][1] *= al1;
            o[mt][2] *= al0;
            o[mt][3] *= al1;
          }
        }
        const float p0 = va ? fast_exp2(x0 - m0) : 0.f, p1 = va ? fast_exp2(x1 - m1) : 0.f;
        const float p2 = vb ? fast_exp2(x2 - m0) : 0.f, p3 = vb ? fast_exp2(x3 - m1) : 0.f;
        l0 += p0 + p2;  // this lane's keys only; summed over the lanes at the end
        l1 += p1 + p3;
        // P^T as the B operand (keys x heads), hi + lo bf16 parts
        const uint32_t bh0 = movmatrix_t(pack_bf16x2(p0, p1)), bh1 = movmatrix_t(pack_bf16x2(p2, p3));
        const uint32_t bl0 = movmatrix_t(pack_bf16x2(bf16_residual(p0), bf16_residual(p1)));
        const uint32_t bl1 = movmatrix_t(pack_bf16x2(bf16_residual(p2), bf16_residual(p3)));
        // O^T += V^T P^T, 16 value dims per block
        const int vr = r0 + (lane & 7) + (lane >> 4) * 8, vc = ((lane >> 3) & 1) * 8;
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
          uint32_t v4[4];
          ldsm_x4_t(v4, tV + swz_off(vr, mt * 16 + vc, kRows));
          mma_m16n8k16(o[mt], v4[0], v4[1], v4[2], v4[3], bh0, bh1);
          mma_m16n8k16(o[mt], v4[0], v4[1], v4[2], v4[3], bl0, bl1);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&empty[st]);
    }
    if (!ok) {
      if (lane == 0) sFail = 1;
      m0 = m1 = kNegInf;
      l0 = l1 = 0.f;
#pragma unroll
      for (int mt = 0; mt < MT; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
    }
#pragma unroll
    for (int off = 4; off < 32; off <<= 1) {
      l0 += __shfl_xor_sync(0xffffffffu, l0, off);
      l1 += __shfl_xor_sync(0xffffffffu, l1, off);
    }

    // ---- the four warps' states into one CTA state, through the ring (free
    // once every attending warp is past its tiles, unless a wait gave up and
    // copies may still land there)
    named_sync(1, kConsumerWarps * 32);
    const bool bad = sFail != 0;
    float* sW = reinterpret_cast<float*>(ring);  // [4][G][D] O
    float* sWml = sW + 4 * G * D;                // [4][G][2] (m, l)
    if (!bad) {
#pragma unroll
      for (int mt = 0; mt < MT; ++mt) {
        if (2 * t < G) {
          sW[(warp * G + 2 * t) * D + mt * 16 + g] = o[mt][0];
          sW[(warp * G + 2 * t) * D + mt * 16 + g + 8] = o[mt][2];
        }
        if (2 * t + 1 < G) {
          sW[(warp * G + 2 * t + 1) * D + mt * 16 + g] = o[mt][1];
          sW[(warp * G + 2 * t + 1) * D + mt * 16 + g + 8] = o[mt][3];
        }
      }
      if (g == 0 && 2 * t < G) {
        sWml[(warp * G + 2 * t) * 2] = m0;
        sWml[(warp * G + 2 * t) * 2 + 1] = l0;
        if (2 * t + 1 < G) {
          sWml[(warp * G + 2 * t + 1) * 2] = m1;
          sWml[(warp * G + 2 * t + 1) * 2 + 1] = l1;
        }
      }
    }
    named_sync(2, kConsumerWarps * 32);
    cluster_wait_acquire();  // every CTA of the cluster has started and armed its receive barrier
    // thread -> (head, 4 dims): the CTA's state for them goes to the owner of those dims
    for (int it = tid; it < G * D / 4; it += kConsumerWarps * 32) {
      const int h = it / (D / 4), d0 = (it % (D / 4)) * 4;
      float mw[kConsumerWarps], lw[kConsumerWarps], M = kNegInf;
#pragma unroll
      for (int w = 0; w < kConsumerWarps; ++w) {
        mw[w] = bad ? kNegInf : sWml[(w * G + h) * 2];
        lw[w] = bad ? 0.f : sWml[(w * G + h) * 2 + 1];
        if (lw[w] > 0.f) M = fmaxf(M, mw[w]);
      }
      float L = 0.f;
      float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
      if (M != kNegInf) {
#pragma unroll
        for (int w = 0; w < kConsumerWarps; ++w) {
          if (lw[w] > 0.f) {
            const float f = fast_exp2(mw[w] - M);
            const float4 v = *reinterpret_cast<const float4*>(sW + (w * G + h) * D + d0);
            L = fmaf(lw[w], f, L);
            acc.x = fmaf(f, v.x, acc.x);
            acc.y = fmaf(f, v.y, acc.y);
            acc.z = fmaf(f, v.z, acc.z);
            acc.w = fmaf(f, v.w, acc.w);
          }
        }
      }
      const int rr = sOwner[d0 >> 4], lo = sLo[d0 >> 4] * 16;
      const uint32_t bar = cluster_map(&recv, rr);
      st_async_v4(cluster_map(rcv_o + ((size_t)s * G + h) * OD + (d0 - lo), rr), acc, bar);
      if (d0 == lo) st_async_v2(cluster_map(rcv_ml + ((size_t)s * G + h) * 2, rr), M, L, bar);
    }

  }

  // ---- local parts (f_hat_E rows, per-head weights, v_new) in place; the
  // other CTAs' states for the owned dims landed
  __syncthreads();
  const bool got_all = mbar_wait(&recv, 0);
  if (!got_all && tid == 0) record_error(a.ws, MKV_ERR_TIMEOUT, u);

  // ---- owner merge (log2 domain): one (head, owned dim) output per thread
  for (int idx = tid; idx < G * own_d; idx += kClThreads) {
    const int h = idx / own_d, j = idx % own_d;
    float2 ml[kMaxSplits];
    float M = has_new ? sSn[h] : kNegInf;
#pragma unroll
    for (int sl = 0; sl < kMaxSplits; ++sl) {
      ml[sl] = sl < S ? *reinterpret_cast<const float2*>(rcv_ml + ((size_t)sl * G + h) * 2) : make_float2(kNegInf, 0.f);
      if (ml[sl].y > 0.f) M = fmaxf(M, ml[sl].x);
    }
    float L = 0.f, O = 0.f;
    if (M != kNegInf) {
#pragma unroll
      for (int sl = 0; sl < kMaxSplits; ++sl) {
        if (ml[sl].y > 0.f) {
          const float w = fast_exp2(ml[sl].x - M);
          L = fmaf(ml[sl].y, w, L);
          O = fmaf(w, rcv_o[((size_t)sl * G + h) * OD + j], O);
        }
      }
      if (has_new) {
        const float w = fast_exp2(sSn[h] - M);
        L += w;
        O = fmaf(w, sVn[j], O);
      }
    }
    const bool have_r = L > 0.f;
    float res, lse2;  // output, log2 of the normaliser
    if (use_m) {
      const float e = sE[h], fh = sF[j * G + h];
      if (have_r) {
        const float a2 = M + fast_log2(L);
        const float top = fmaxf(a2, e);
        const float wr = fast_exp2(a2 - top), we = fast_exp2(e - top);
        const float inv = fast_rcp(wr + we);
        res = (wr * inv) * (O * fast_rcp(L)) + (we * inv) * fh;
        lse2 = top + fast_log2(wr + we);
      } else {
        res = fh;
        lse2 = e;
      }
    } else {
      if (!have_r && j == 0) record_error(a.ws, MKV_ERR_INVALID_ARG, u);
      res = have_r ? O * fast_rcp(L) : 0.f;
      lse2 = have_r ? M + fast_log2(L) : kNegInf;
    }
    const int dim = mlo * 16 + j;
    a.out[((size_t)u * G + h) * D + dim] = res;
    if (a.lse != nullptr && dim == 0) a.lse[(size_t)u * G + h] = lse2 * kLn2;
  }

  if (producer && lane == 0) {
    if (s == 0 && has_new) {  // the row itself was written by CTA S - 1
      if (len0 + 1 > a.cap) {
        record_error(a.ws, MKV_ERR_CAPACITY, u);
      } else {
        a.pos[(size_t)u * a.cap + len0] = seen0;
        st_hint(a.seen + u, seen0 + 1, pol_keep);
        st_hint(a.len + u, len0 + 1, pol_keep);
      }
    }
    if (sFail) {
      record_error(a.ws, MKV_ERR_TIMEOUT, u);
      // drain the copies still owed to this CTA before its shared memory is
      // released: the last tile issued into each stage
      for (int i = max(0, issued - NST); i < issued; ++i) (void)mbar_wait(&full[i % NST], (i / NST) & 1);
    }
  }
}

template <int D, int G, bool C16, bool EARLY>
int cl_active_clusters(int S) {
  constexpr int kMaxDev = 64;
  static std::mutex mu;
  static int known[kMaxDev][9] = {};
  int dev = 0;
  if (S < 1 || S > 8 || cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return 0;
  std::lock_guard<std::mutex> lock(mu);
  if (known[dev][S] == 0) {
    const size_t smem = cl_smem_bytes(D, G, S);
    int n = 0;
    cudaError_t e = cudaFuncSetAttribute(decode_cl_kernel<D, G, C16, EARLY, false>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e == cudaSuccess) {
      cudaLaunchConfig_t cfg{};
      cfg.gridDim = dim3(S, 1, 1);
      cfg.blockDim = dim3(kClThreads, 1, 1);
      cfg.dynamicSmemBytes = smem;
      cudaLaunchAttribute at[1];
      at[0].id = cudaLaunchAttributeClusterDimension;
      at[0].val.clusterDim.x = S;
      at[0].val.clusterDim.y = 1;
      at[0].val.clusterDim.z = 1;
      cfg.attrs = at;
      cfg.numAttrs = 1;
      e = cudaOccupancyMaxActiveClusters(&n, decode_cl_kernel<D, G, C16, EARLY, false>, &cfg);
    }
    if (e != cudaSuccess) {
      (void)cudaGetLastError();
      n = 0;
    }
    known[dev][S] = n > 0 ? n : -1;
  }
  return known[dev][S];
}

template <int D, int G, bool C16, bool EARLY, bool CS>
cudaError_t launch_cl(const DecodeArgs& args, cudaStream_t stream) {
  DecodeArgs a = args;
  a.S = a.S_cl;
  a.polls = pipeline_poll_limit();
  const size_t smem = cl_smem_bytes(D, G, a.S);
  cudaError_t e = cudaFuncSetAttribute(decode_cl_kernel<D, G, C16, EARLY, CS>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const uint64_t rows = (uint64_t)a.batch * a.n_kv * a.cap;  // the cache slabs of all units as one matrix
  CUtensorMap tmK, tmV;
  if (!encode_tmap_bf16(&tmK, a.K, D, rows, (uint64_t)D * 2, 64, kRows) ||
      !encode_tmap_bf16(&tmV, a.V, D, rows, (uint64_t)D * 2, 64, kRows))
    return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(a.S, a.n_kv, a.batch);
  cfg.blockDim = dim3(kClThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute at[2];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  at[1].id = cudaLaunchAttributeClusterDimension;
  at[1].val.clusterDim.x = a.S;
  at[1].val.clusterDim.y = 1;
  at[1].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, decode_cl_kernel<D, G, C16, EARLY, CS>, a, tmK, tmV);
}

// C as fp32, as its bf16 copy, or in the operand form (validation rejects both copies at once)
template <int D, int G>
cudaError_t launch_cl_dg(const DecodeArgs& a, cudaStream_t stream) {
  if (a.early) {
    if (a.C16 != nullptr) return launch_cl<D, G, true, true, false>(a, stream);
    return a.Cs != nullptr ? launch_cl<D, G, false, true, true>(a, stream) : launch_cl<D, G, false, true, false>(a, stream);
  }
  if (a.C16 != nullptr) return launch_cl<D, G, true, false, false>(a, stream);
  return a.Cs != nullptr ? launch_cl<D, G, false, false, true>(a, stream) : launch_cl<D, G, false, false, false>(a, stream);
}

template <int D, int G>
int cl_active_dg(int S) {
  return cl_active_clusters<D, G, false, false>(S);
}

}  // namespace

// Split count of the cluster kernel: at most 8 (a portable cluster), one
// 64-row tile per CTA at most as many as the capacity needs, and at most one
// CTA per SM when the launch is a link of a layer chain (early_load), so
// that the next layer's CTAs are resident and load their tiles while this
// launch runs; two per SM otherwise.  0 when no cluster of that size fits.
int decode_cluster_splits(const mkv_geom& g, int32_t capacity, int num_sms, int early) {
  const long units = (long)g.batch * g.n_kv_heads;
  const long tiles = ((long)capacity + 1 + kRows - 1) / kRows;
  const long slots = (early ? 1L : 2L) * num_sms;
  long S = std::min<long>(std::min(8L, tiles), std::max(1L, slots / units));
  if (S < 1) S = 1;
  int n = 0;
#define MKV_CLA_CASE(D_, G_) \
  if (g.head_dim == D_ && g.group == G_) n = cl_active_dg<D_, G_>(static_cast<int>(S));
  MKV_CLA_CASE(128, 1)
  MKV_CLA_CASE(128, 2)
  MKV_CLA_CASE(128, 4)
  MKV_CLA_CASE(128, 8)
  MKV_CLA_CASE(64, 1)
  MKV_CLA_CASE(64, 2)
  MKV_CLA_CASE(64, 4)
  MKV_CLA_CASE(64, 8)
#undef MKV_CLA_CASE
  return n > 0 ? static_cast<int>(S) : 0;
}

cudaError_t launch_decode_cluster(const DecodeArgs& a, int head_dim, int group, cudaStream_t stream) {
#define MKV_CL_CASE(D_, G_) \
  if (head_dim == D_ && group == G_) return launch_cl_dg<D_, G_>(a, stream);
  MKV_CL_CASE(128, 1)
  MKV_CL_CASE(128, 2)
  MKV_CL_CASE(128, 4)
  MKV_CL_CASE(128, 8)
  MKV_CL_CASE(64, 1)
  MKV_CL_CASE(64, 2)
  MKV_CL_CASE(64, 4)
  MKV_CL_CASE(64, 8)
#undef MKV_CL_CASE
  return cudaErrorInvalidValue;
}

}  // namespace mkv
