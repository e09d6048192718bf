// Prefill compression (Sec. 5.1 SnapKV protocol with the moment filter of
// Sec. 4.2, read as two data-parallel selection stages).
//
// Launch sequence per call (one stream):
//   stats_tc  (chunk, unit)  window logits Q_obs K^T on the tensor cores ->
//                            online (max, sum) of each causal window row; the
//                            covariance V^T K accumulated in TMEM and the column
//                            sums -> the chunk's centred moments
//   scores_tc (chunk, unit)  logits again (token-major) -> s_t = sum over rows
//                            of exp(l - m_row) / l_row, pooled
//   select    (8-CTA cluster per unit) R0 = protected + top-k(s): radix select
//                            with 8-bit digits, histograms summed through
//                            distributed shared memory, ties to the lower
//                            position; R0's rows gathered densely
//   stats_tc  (chunk, unit)  moments of the gathered R0 rows (no logits)
//   finalize  (rows, unit)   M0 = moments(all) - moments(R0) (Chan merges); the
//                            all-token record is merged once and kept
//   residual_tc (chunk, unit) Y = K C0'^T on the tensor cores (C0' split into
//                            three bf16 parts) -> score2 = s_t ||v - mu_v0 - scale y||
//   select    (cluster, unit) R = protected + top-k(score2), gathered into the cache
//   stats_tc  (chunk, unit)  moments of the retained rows
//   finalize  (rows, unit)   moments of E = all \ R -> caller's mkv_moments
//
// With the budget shared by the KV heads of a batch item (adaptive), each
// select ranks the (head, position) pairs of the batch item together: a
// per-unit select first keeps each head's own top k as candidates (the joint
// top k lies among them) when that prunes at least half the pairs, then one
// cluster per batch item ranks the candidates.  gather_kernel copies the
// unequal per-head row sets, and stats_tc / gather_kernel take a grid over
// each batch item's actual 128-row tiles.
//
// The tensor-core kernels are warp-specialised: warp 0 issues the TMA copies
// (3-D tensor maps over per-unit slabs: rows past a unit's end read as zeros),
// warp 1 owns TMEM and issues tcgen05.mma, and the other warps run the
// epilogue (two groups of four in stats_tc, scores_tc and residual_tc);
// stages hand over through mbarriers whose waits are all bounded.  Head dims
// below 128 use the same 128-wide MMAs: the missing 64-column box is
// zero-filled.
#include <algorithm>
#include <cooperative_groups.h>

#include "common.cuh"
#include "kernels.h"
#include "tc.cuh"

namespace cg = cooperative_groups;

namespace mkv {

namespace {

constexpr int kTok = 128;                   // tokens per tile
constexpr int kDP = 128;                    // padded head dim of every MMA
constexpr int kTileBytes = kTok * kDP * 2;  // one [128 x 128] bf16 tile: 2 boxes of 16 KB
constexpr int kBoxBytes = kTok * 128;
// stats_tc: two epilogue groups of 4 warps (2..5 and 6..9), each taking half
// of a tile's tokens, so that two warps per scheduler share the softmax work
constexpr int kStatsThreads = 320;
constexpr int kSelThreads = 1024;
constexpr int kPF = 0;  // tiles prefetched into L2 ahead of the one being loaded (0: none)
constexpr unsigned kFull = 0xffffffffu;

struct Layout {
  int D, G, W, RW, RWb;  // head dim, group, window, window rows = G*W, 128-row blocks of them
  int T, B;
  int hs;    // units per selection group: 1, or the KV heads of a batch item (adaptive budget)
  int Bcap;  // rows of each unit's gathered slab: B, or the adaptive maximum rounded up to kTok
  int Tc;    // joint selection entries per unit: T, or the length of its candidate list
  int units, n_chunks, chunk;
  size_t rec;         // floats per moment record: 4 + 2D + D*D (padded)
  float* rowpart;     // [units][n_chunks][RW][2]  (max in log2 units, sum)
  float* mpart;       // [units][n_chunks][rec]    all-token chunk moments
  float* rpart;       // [units][n_rchunks][rec]   retained-set chunk moments
  int n_rchunks;      // chunks of kTok retained rows
  float* s;           // [units][T]
  float* s2;          // [units][T]
  int32_t* idx;       // [units / hs][hs * B] selection lists (h * T + t), ascending
  int32_t* cnt;       // [units] rows each unit retains
  int32_t* cand;      // [units][Tc] per-unit candidates of a joint selection (when Tc < T)
  int32_t* hbeg;      // [units] first slot of each unit in idx
  int32_t* tile0;     // [units / hs][hs + 1] first retained-row tile of each unit in its group (joint)
  int gtiles;         // bound on a group's retained-row tiles (joint)
  __nv_bfloat16* gK;  // [units][Bcap][D] rows of R0
  __nv_bfloat16* gV;
  float* m0;    // [units][rec] moments of E0
  float* mall;  // [units][rec] moments of all tokens (the merged chunk records)
};

__host__ __device__ inline size_t rec_floats(int D) { return align_up(4 + 2 * (size_t)D + (size_t)D * D, 4); }

__host__ __device__ __forceinline__ int protected_count(int T, int W, int sink, int keep_window) {
  const int s = sink < T ? sink : T;
  const int w = keep_window ? (W < T ? W : T) : 0;
  const int overlap = s - (T - w) > 0 ? s - (T - w) : 0;
  return s + w - overlap;
}

Layout make_layout(const mkv_geom& g, int T, int B, int W, int sink, int keep_window, int adaptive,
                   int num_sms) {
  Layout L{};
  L.hs = 1;
  L.Bcap = B;
  L.Tc = T;
  if (adaptive && T > B) {  // a unit keeps its protected rows plus up to every joint selection
    const long prot = protected_count(T, W, sink, keep_window);
    const long most = std::min<long>(T, (long)g.n_kv_heads * (B - prot) + prot);
    L.hs = g.n_kv_heads;
    L.Bcap = static_cast<int>((most + kTok - 1) / kTok * kTok);
    // every pair of the joint top k is in its own head's top k, so a first
    // per-unit selection of those (`most` rows with the protected ones)
    // leaves the joint one fewer entries when they are well below T
    if (2 * most <= T) L.Tc = static_cast<int>(most);
    // sum_h ceil(c_h / kTok) with sum_h c_h = hs * B
    L.gtiles = static_cast<int>(((long)L.hs * B + (long)L.hs * (kTok - 1)) / kTok);
  }
  L.D = g.head_dim;
  L.G = g.group;
  L.W = W;
  L.RW = g.group * W;
  L.RWb = (L.RW + 127) / 128;
  L.T = T;
  L.B = B;
  L.units = g.batch * g.n_kv_heads;
  long per = num_sms / L.units;  // one resident CTA per SM: fill the machine once
  const long tiles = (T + kTok - 1) / kTok;
  if (per < 1) per = 1;
  if (per > tiles) per = tiles;
  L.chunk = static_cast<int>(((tiles + per - 1) / per) * kTok);
  L.n_chunks = (T + L.chunk - 1) / L.chunk;
  L.rec = rec_floats(L.D);
  L.n_rchunks = (L.Bcap + kTok - 1) / kTok;
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
  L.rpart = reinterpret_cast<float*>(take(U * L.n_rchunks * L.rec * sizeof(float)));
  L.s = reinterpret_cast<float*>(take(U * (size_t)L.T * sizeof(float)));
  L.s2 = reinterpret_cast<float*>(take(U * (size_t)L.T * sizeof(float)));
  L.idx = reinterpret_cast<int32_t*>(take(U * (size_t)L.B * sizeof(int32_t)));
  L.cnt = reinterpret_cast<int32_t*>(take(U * sizeof(int32_t)));
  L.cand = L.Tc < L.T ? reinterpret_cast<int32_t*>(take(U * (size_t)L.Tc * sizeof(int32_t))) : nullptr;
  L.hbeg = reinterpret_cast<int32_t*>(take(U * sizeof(int32_t)));
  L.tile0 = reinterpret_cast<int32_t*>(take((U / L.hs) * (size_t)(L.hs + 1) * sizeof(int32_t)));
  L.gK = reinterpret_cast<__nv_bfloat16*>(take(U * (size_t)L.Bcap * L.D * 2));
  L.gV = reinterpret_cast<__nv_bfloat16*>(take(U * (size_t)L.Bcap * L.D * 2));
  L.m0 = reinterpret_cast<float*>(take(U * L.rec * sizeof(float)));
  L.mall = reinterpret_cast<float*>(take(U * L.rec * sizeof(float)));
  return off;
}

__device__ __forceinline__ bool is_protected(int t, int T, int W, int sink, int keep_window) {
  return t < sink || (keep_window && t >= T - W);
}

__device__ __forceinline__ void epi_sync() { asm volatile("bar.sync 1, 128;" ::: "memory"); }
// whether v holds in all 128 threads of the first epilogue group (barrier 1)
__device__ __forceinline__ bool epi_all(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\tsetp.ne.u32 p, %1, 0;\n\tbar.red.and.pred q, 1, 128, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"((uint32_t)v)
      : "memory");
  return r != 0;
}

// Pipeline wait that gives up after `polls` polls: records the timeout once
// and raises the CTA's abort flag so that no other role waits on.
__device__ __forceinline__ bool pwait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, void* ws, int u,
                                      uint32_t polls) {
  if (*abort_flag) return false;
  if (mbar_wait(bar, parity, polls)) return true;
  *abort_flag = 1;
  record_error(ws, MKV_ERR_TIMEOUT, u);
  return false;
}

// After an abort, before a CTA frees its tensor memory and exits: wait (with
// the full poll limit) for the last tile copy issued into each of the kS
// stages, for the window-query copy if one was issued, and for the MMA
// thread's final commit (every MMA it issued has completed, so none still
// reads shared memory or writes TMEM).  `issued` tiles went out in order,
// tile i into stage i % kS.
__device__ __forceinline__ void drain_after_abort(uint64_t* full, int kS, int issued, uint64_t* qfull,
                                                  uint64_t* mma_done) {
  for (int st = 0; st < kS; ++st) {
    const int last = issued - 1 - ((issued - 1 - st) % kS + kS) % kS;  // largest i < issued with i % kS == st
    if (last >= 0 && last % kS == st) (void)mbar_wait(&full[st], (last / kS) & 1);
  }
  if (qfull != nullptr) (void)mbar_wait(qfull, 0);
  (void)mbar_wait(mma_done, 0);
}

struct TcArgs {
  int n_rows;  // rows of each unit's slab that take part
  const int32_t* rows_u;  // optional per-unit row counts (<= n_rows) that replace n_rows
  const int32_t* tile0;   // optional [groups][hs + 1]: grid (tiles of a group, groups), as in gather_kernel
  int hs;
  int chunk;   // rows per CTA (multiple of kTok)
  int n_chunks;
  int D, RW, RWb, W, T, causal, sink, keep_window, pool;
  float qscale;  // scale * log2(e)
  float tau;
  float* rowpart;
  float* mrec;  // moment records, [units][n_chunks][rec]
  const float* s_in;
  float* s_out;
  float* diag;
  const float* m0;
  void* ws;
  uint32_t polls;  // poll limit of the pipeline waits
};

// --------------------------------------------------------------- stats_tc
// LOGITS = 1: window-row statistics and chunk moments of the prompt;
// LOGITS = 0: moments only (a dense row set).
template <int LOGITS>
__global__ void __launch_bounds__(kStatsThreads, 1)
    stats_tc(const TcArgs p, const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
             const __grid_constant__ CUtensorMap tmQ) {
  // without logits (moments of a gathered row set, one tile per CTA): one
  // stage, no Q, and half the TMEM, so that several CTAs share an SM
  constexpr int kS = LOGITS ? 2 : 1;
  constexpr uint32_t kTmemCols = LOGITS ? 512 : 256;
  constexpr int cS = LOGITS ? 256 : 0, cSum = LOGITS ? 384 : 128;  // TMEM columns of V^T K and the sums
  extern __shared__ __align__(1024) uint8_t smraw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023));
  uint8_t* sK = sm;                        // [kS][128 x 128]
  uint8_t* sV = sm + kS * kTileBytes;      // [kS][128 x 128]
  uint8_t* sQ = sm + 2 * kS * kTileBytes;  // [2 boxes][RWb*128 rows][128 B]
  uint8_t* sOnes = sQ + (LOGITS ? 2 * 2 * kBoxBytes : 0);  // [2 boxes][16 rows][128 B] of bf16 1.0
  __shared__ __align__(8) uint64_t full[kS], empty[kS], lfull, lempty, qfull, sdone;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag, s_issued;
  __shared__ float sum_k[kDP], sum_v[kDP];
  __shared__ float s_m1[2][128], s_l1[2][128];  // the second epilogue group's row stats

  int chunk = blockIdx.x, u = blockIdx.y;
  if (!LOGITS && p.tile0 != nullptr) {  // the group's tiles, unit by unit
    const int32_t* t0 = p.tile0 + (size_t)blockIdx.y * (p.hs + 1);
    if (chunk >= t0[p.hs]) return;
    int h = 0;
    while (h + 1 < p.hs && t0[h + 1] <= chunk) ++h;
    u = blockIdx.y * p.hs + h;
    chunk -= t0[h];
  }
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int t_begin = chunk * p.chunk;
  const int n_rows = (!LOGITS && p.rows_u != nullptr) ? p.rows_u[u] : p.n_rows;
  const int t_end = min(n_rows, t_begin + p.chunk);
  const int n_tiles = (max(0, t_end - t_begin) + kTok - 1) / kTok;
  const int RWb = p.RWb;
  volatile int* abrt = &abort_flag;
  if (!LOGITS && n_tiles == 0) {  // a chunk past this unit's rows: an empty record (n = 0, zero means)
    float* rec = p.mrec + ((size_t)u * p.n_chunks + chunk) * rec_floats(p.D);
    for (int i = tid; i < 4 + 2 * p.D; i += kStatsThreads) rec[i] = 0.f;
    return;
  }

  if (tid == 0) {
    for (int i = 0; i < kS; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);  // the stage is free once its MMAs have completed
    }
    mbar_init(&lfull, 1);
    mbar_init(&lempty, 8);
    mbar_init(&qfull, 1);
    mbar_init(&sdone, 1);
    abort_flag = 0;
    s_issued = 0;
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc(&tmem_base, kTmemCols);
  if (warp >= 2 && warp < 6) {  // the ones operand of the column sums K^T 1 and V^T 1
    for (int i = tid - 64; i < 2 * 16 * 128 / 16; i += 128)
      reinterpret_cast<uint4*>(sOnes)[i] = make_uint4(0x3F803F80u, 0x3F803F80u, 0x3F803F80u, 0x3F803F80u);
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = tmem_base;

  if (warp == 0) {
    if (lane == 0) {  // ---- producer
      if (LOGITS) {
        mbar_arrive_expect_tx(&qfull, 2u * RWb * kBoxBytes);
        for (int bx = 0; bx < 2; ++bx) tma_load_3d(sQ + bx * RWb * kBoxBytes, &tmQ, bx * 64, 0, u, &qfull);
      }
      for (int i = 0; i < min(kPF, n_tiles); ++i)
        for (int bx = 0; bx < 2; ++bx) {
          tma_prefetch_3d(&tmK, bx * 64, t_begin + i * kTok, u);
          tma_prefetch_3d(&tmV, bx * 64, t_begin + i * kTok, u);
        }
      for (int i = 0; i < n_tiles; ++i) {
        const int s = i % kS, j = i / kS;
        if (kPF > 0 && i + kPF < n_tiles)
          for (int bx = 0; bx < 2; ++bx) {
            tma_prefetch_3d(&tmK, bx * 64, t_begin + (i + kPF) * kTok, u);
            tma_prefetch_3d(&tmV, bx * 64, t_begin + (i + kPF) * kTok, u);
          }
        if (j >= 1 && !pwait(&empty[s], (j - 1) & 1, abrt, p.ws, u, p.polls)) break;
        mbar_arrive_expect_tx(&full[s], 2u * kTileBytes);
        for (int bx = 0; bx < 2; ++bx) {
          tma_load_3d(sK + s * kTileBytes + bx * kBoxBytes, &tmK, bx * 64, t_begin + i * kTok, u, &full[s]);
          tma_load_3d(sV + s * kTileBytes + bx * kBoxBytes, &tmV, bx * 64, t_begin + i * kTok, u, &full[s]);
        }
        s_issued = i + 1;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {  // ---- MMA issuer
      const uint32_t idL = idesc_bf16(128, 128, 0, 0);  // logits: rows x tokens, both K-major
      const uint32_t idS = idesc_bf16(128, 128, 1, 1);  // V^T K: both MN-major (reduction over tokens)
      const uint32_t id1 = idesc_bf16(128, 16, 1, 0);   // X^T 1: X MN-major, ones K-major
      const uint32_t aQ = smem_addr(sQ), a1 = smem_addr(sOnes);
      const bool ok = !LOGITS || pwait(&qfull, 0, abrt, p.ws, u, p.polls);
      for (int i = 0; ok && i < n_tiles; ++i) {
        const int s = i % kS, j = i / kS;
        if (!pwait(&full[s], j & 1, abrt, p.ws, u, p.polls)) break;
        tc_fence_after();
        const uint32_t aK = smem_addr(sK + s * kTileBytes), aV = smem_addr(sV + s * kTileBytes);
        if (LOGITS) {
          if (i >= 1 && !pwait(&lempty, (i - 1) & 1, abrt, p.ws, u, p.polls)) break;
          tc_fence_after();
          for (int rb = 0; rb < RWb; ++rb)
            for (int kk = 0; kk < 8; ++kk) {
              const uint64_t dq =
                  sdesc_sw128(aQ + (kk >> 2) * RWb * kBoxBytes + rb * kBoxBytes + (kk & 3) * 32, 16, 1024);
              const uint64_t dk = sdesc_sw128(aK + (kk >> 2) * kBoxBytes + (kk & 3) * 32, 16, 1024);
              umma_bf16(tm + rb * 128, dq, dk, idL, kk > 0 ? 1u : 0u);
            }
          umma_commit(&lfull);
        }
        for (int kk = 0; kk < 8; ++kk) {
          const uint64_t dv = sdesc_sw128(aV + kk * 2048, kBoxBytes, 1024);
          const uint64_t dk = sdesc_sw128(aK + kk * 2048, kBoxBytes, 1024);
          const uint64_t d1 = sdesc_sw128(a1 + (kk >> 2) * 2048 + (kk & 3) * 32, 16, 1024);
          const uint32_t acc = (i > 0 || kk > 0) ? 1u : 0u;
          umma_bf16(tm + cS, dv, dk, idS, acc);
          umma_bf16(tm + cSum, dk, d1, id1, acc);       // column sums of K (lane = key dim)
          umma_bf16(tm + cSum + 16, dv, d1, id1, acc);  // column sums of V (lane = value dim)
        }
        umma_commit(&empty[s]);
      }
      umma_commit(&sdone);
    }
  } else {
    // ---- epilogue: group 0 = warps 2..5 (tokens 0..63 of a tile), group 1 =
    // warps 6..9 (tokens 64..127); TMEM lane quarter qd = warp % 4
    const int grp = (warp - 2) >> 2;
    const int et = tid - 64 - grp * 128, qd = warp & 3;
    const uint32_t lane_base = static_cast<uint32_t>(qd * 32) << 16;
    float m[2] = {-INFINITY, -INFINITY}, l[2] = {0.f, 0.f};
    int tmax_vis[2];
    for (int rb = 0; rb < 2; ++rb) {
      const int r = rb * 128 + qd * 32 + lane;  // window row of this thread
      tmax_vis[rb] = p.causal ? p.T - p.W + r % p.W : 0x7fffffff;
    }
    const int t_safe = p.causal ? p.T - p.W : 0x7fffffff;  // tokens every window row sees
    for (int i = 0; LOGITS && i < n_tiles; ++i) {
      if (!pwait(&lfull, i & 1, abrt, p.ws, u, p.polls)) break;
      tc_fence_after();
      const int tt0 = t_begin + i * kTok;
      const bool fast = tt0 + kTok <= t_end && tt0 + kTok - 1 <= t_safe;  // no masking in this tile
      // rb runs over a constant range (guarded by RWb), so that m, l and
      // tmax_vis stay in registers
#pragma unroll
      for (int rb = 0; rb < 2; ++rb) {
        if (rb >= RWb) break;
        for (int c0 = grp * 64; c0 < grp * 64 + 64; c0 += 32) {
          float x[32];
          tmem_ld32(tm + lane_base + rb * 128 + c0, x);
          const int t0 = tt0 + c0;
          float mx = -INFINITY;
          if (fast) {
#pragma unroll
            for (int jj = 0; jj < 32; ++jj) {
              x[jj] *= p.qscale;
              mx = fmaxf(mx, x[jj]);
            }
          } else {
#pragma unroll
            for (int jj = 0; jj < 32; ++jj) {
              const int t = t0 + jj;
              x[jj] = (t < t_end && t <= tmax_vis[rb]) ? x[jj] * p.qscale : -INFINITY;
              mx = fmaxf(mx, x[jj]);
            }
          }
          {
            const float mn = fmaxf(m[rb], mx);
            if (mn != -INFINITY) {
              float acc = 0.f;
#pragma unroll
              for (int jj = 0; jj < 32; ++jj) acc += fast_exp2(x[jj] - mn);
              l[rb] = l[rb] * fast_exp2(m[rb] - mn) + acc;
              m[rb] = mn;
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&lempty);
    }
    if (LOGITS) {  // merge the two groups' (max, sum) of each row
      if (grp == 1)
#pragma unroll
        for (int rb = 0; rb < 2; ++rb) {
          if (rb < RWb) {
            s_m1[rb][qd * 32 + lane] = m[rb];
            s_l1[rb][qd * 32 + lane] = l[rb];
          }
        }
      asm volatile("bar.sync 2, 256;" ::: "memory");
      if (grp == 0)
#pragma unroll
        for (int rb = 0; rb < 2; ++rb) {
          if (rb >= RWb) break;
          const int r = rb * 128 + qd * 32 + lane;
          const float m1 = s_m1[rb][qd * 32 + lane], l1 = s_l1[rb][qd * 32 + lane];
          const float M = fmaxf(m[rb], m1);
          float L = 0.f;
          if (M != -INFINITY) {
            if (m[rb] != -INFINITY) L += l[rb] * fast_exp2(m[rb] - M);
            if (m1 != -INFINITY) L += l1 * fast_exp2(m1 - M);
          }
          if (r < p.RW) {
            float* rp = p.rowpart + (((size_t)u * p.n_chunks + chunk) * p.RW + r) * 2;
            rp[0] = M;
            rp[1] = L;
          }
        }
    }
    if (grp == 0) {
    // uniform over the group: after an abort the MMAs may still write TMEM,
    // so it is not read and the chunk's record is left empty
    const bool got = epi_all(pwait(&sdone, 0, abrt, p.ws, u, p.polls));
    float* rec = p.mrec + ((size_t)u * p.n_chunks + chunk) * rec_floats(p.D);
    const float nc = got ? static_cast<float>(max(0, t_end - t_begin)) : 0.f;
    if (got) {
    tc_fence_after();
    {
      float x[32];
      tmem_ld32(tm + lane_base + cSum, x);  // [0]: sum of K's column (this lane), [16]: of V's
      sum_k[qd * 32 + lane] = x[0];
      sum_v[qd * 32 + lane] = x[16];
    }
    epi_sync();
    const float inv_nc = nc > 0.f ? 1.f / nc : 0.f;
    const int a = qd * 32 + lane;  // value dim = TMEM lane
    // centred co-moment rows staged 32 columns at a time through the (now
    // free) K stage, so that the record is written in coalesced rows
    float* stg = reinterpret_cast<float*>(sK);  // [128][33]
    for (int c0 = 0; c0 < kDP; c0 += 32) {
      float srow[32];
      tmem_ld32(tm + lane_base + cS + c0, srow);
#pragma unroll
      for (int jj = 0; jj < 32; ++jj) stg[a * 33 + jj] = srow[jj] - sum_v[a] * sum_k[c0 + jj] * inv_nc;
      epi_sync();
      if (nc > 0.f)
        for (int idx = et; idx < 128 * 32; idx += 128) {
          const int r = idx >> 5, c = c0 + (idx & 31);
          if (r < p.D && c < p.D) rec[4 + 2 * p.D + (size_t)r * p.D + c] = stg[r * 33 + (idx & 31)];
        }
      epi_sync();
    }
    if (a < p.D) {
      rec[4 + a] = nc > 0.f ? sum_k[a] / nc : 0.f;
      rec[4 + p.D + a] = nc > 0.f ? sum_v[a] / nc : 0.f;
    }
    } else if (et < 4 + 2 * p.D) {
      rec[et] = 0.f;  // an empty record: n = 0, zero means
    }
    if (et == 0) rec[0] = nc;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (abort_flag) {  // uniform: every role has left its loop
    if (tid == 0) drain_after_abort(full, kS, s_issued, LOGITS ? &qfull : nullptr, &sdone);
    __syncthreads();
  }
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tm, kTmemCols);
  }
}

// -------------------------------------------------------------- scores_tc
__global__ void __launch_bounds__(kStatsThreads, 1)
    scores_tc(const TcArgs p, const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmQ) {
  constexpr int kS = 3;
  extern __shared__ __align__(1024) uint8_t smraw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023));
  uint8_t* sK = sm;                    // [kS][128 x 128]
  uint8_t* sQ = sm + kS * kTileBytes;  // [2 boxes][RWb*128][128 B]
  __shared__ __align__(8) uint64_t full[kS], empty[kS], lfull[2], lempty[2], qfull, mma_done;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag, s_issued;
  __shared__ __align__(16) float s_b[256];  // log2(1 / l_r) - m_r (-inf for padding rows)
  __shared__ int s_wi[256];                   // window index of row r (r mod W)

  const int chunk = blockIdx.x, u = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int t_begin = chunk * p.chunk;
  const int t_end = min(p.n_rows, t_begin + p.chunk);
  const int n_tiles = (max(0, t_end - t_begin) + kTok - 1) / kTok;
  const int RWb = p.RWb, RWp = RWb * 128;
  volatile int* abrt = &abort_flag;

  if (tid == 0) {
    for (int i = 0; i < kS; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&lfull[i], 1);
      mbar_init(&lempty[i], 4);
    }
    mbar_init(&qfull, 1);
    mbar_init(&mma_done, 1);
    abort_flag = 0;
    s_issued = 0;
    mbar_fence_init();
  }
  if (warp == 1) tmem_alloc(&tmem_base, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = tmem_base;

  if (warp == 0) {
    if (lane == 0) {
      mbar_arrive_expect_tx(&qfull, 2u * RWb * kBoxBytes);
      for (int bx = 0; bx < 2; ++bx) tma_load_3d(sQ + bx * RWb * kBoxBytes, &tmQ, bx * 64, 0, u, &qfull);
      for (int i = kS; i < min(kS + kPF, n_tiles); ++i)
        for (int bx = 0; bx < 2; ++bx) tma_prefetch_3d(&tmK, bx * 64, t_begin + i * kTok, u);
      for (int i = 0; i < n_tiles; ++i) {
        const int s = i % kS, j = i / kS;
        if (kPF > 0 && i + kS + kPF < n_tiles)
          for (int bx = 0; bx < 2; ++bx) tma_prefetch_3d(&tmK, bx * 64, t_begin + (i + kS + kPF) * kTok, u);
        if (j >= 1 && !pwait(&empty[s], (j - 1) & 1, abrt, p.ws, u, p.polls)) break;
        mbar_arrive_expect_tx(&full[s], kTileBytes);
        for (int bx = 0; bx < 2; ++bx)
          tma_load_3d(sK + s * kTileBytes + bx * kBoxBytes, &tmK, bx * 64, t_begin + i * kTok, u, &full[s]);
        s_issued = i + 1;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t id = idesc_bf16(128, RWp, 0, 0);  // tokens x window rows, both K-major
      const uint32_t aQ = smem_addr(sQ);
      const bool ok = pwait(&qfull, 0, abrt, p.ws, u, p.polls);
      for (int i = 0; ok && i < n_tiles; ++i) {
        const int s = i % kS, j = i / kS, b = i & 1;
        if (!pwait(&full[s], j & 1, abrt, p.ws, u, p.polls)) break;
        if (i >= 2 && !pwait(&lempty[b], ((i >> 1) - 1) & 1, abrt, p.ws, u, p.polls)) break;
        tc_fence_after();
        const uint32_t aK = smem_addr(sK + s * kTileBytes);
        for (int kk = 0; kk < 8; ++kk) {
          const uint64_t dk = sdesc_sw128(aK + (kk >> 2) * kBoxBytes + (kk & 3) * 32, 16, 1024);
          const uint64_t dq = sdesc_sw128(aQ + (kk >> 2) * RWb * kBoxBytes + (kk & 3) * 32, 16, 1024);
          umma_bf16(tm + b * 256, dk, dq, id, kk > 0 ? 1u : 0u);
        }
        umma_commit(&lfull[b]);
        umma_commit(&empty[s]);
      }
      umma_commit(&mma_done);  // every MMA issued has completed
    }
  } else {
    // two epilogue groups (warps 2..5 and 6..9) take alternate tiles; group g
    // always reads TMEM buffer g
    const int grp = (warp - 2) >> 2, qd = warp & 3;
    const uint32_t lane_base = static_cast<uint32_t>(qd * 32) << 16;
    // merged row statistics of every window row
    for (int r = tid - 64; r < RWp; r += 256) {
      float M = -INFINITY, Lsum = 0.f;
      if (r < p.RW) {
        for (int c = 0; c < p.n_chunks; ++c)
          M = fmaxf(M, p.rowpart[(((size_t)u * p.n_chunks + c) * p.RW + r) * 2]);
        if (M != -INFINITY)
          for (int c = 0; c < p.n_chunks; ++c) {
            const float* rp = p.rowpart + (((size_t)u * p.n_chunks + c) * p.RW + r) * 2;
            if (rp[0] != -INFINITY) Lsum += rp[1] * fast_exp2(rp[0] - M);
          }
      }
      s_b[r] = (Lsum > 0.f) ? -log2f(Lsum) - M : -INFINITY;
      s_wi[r] = r % p.W;
    }
    asm volatile("bar.sync 1, 256;" ::: "memory");
    const int t_safe = p.causal ? p.T - p.W : 0x7fffffff;  // tokens every window row sees
    for (int i = grp; i < n_tiles; i += 2) {
      const int b = i & 1;
      if (!pwait(&lfull[b], (i >> 1) & 1, abrt, p.ws, u, p.polls)) break;
      tc_fence_after();
      const int t = t_begin + i * kTok + qd * 32 + lane;  // token of this thread (TMEM lane)
      const bool fast = t <= t_safe;  // every window row sees this token
      float acc = 0.f;
      for (int c0 = 0; c0 < RWp; c0 += 32) {
        float x[32];
        tmem_ld32(tm + lane_base + b * 256 + c0, x);
        if (fast) {  // p = 2^(x qscale + b_r); padding rows have b_r = -inf
#pragma unroll
          for (int jj = 0; jj < 32; jj += 4) {
            const float4 b4 = *reinterpret_cast<const float4*>(s_b + c0 + jj);
            acc += fast_exp2(fmaf(x[jj], p.qscale, b4.x)) + fast_exp2(fmaf(x[jj + 1], p.qscale, b4.y)) +
                   fast_exp2(fmaf(x[jj + 2], p.qscale, b4.z)) + fast_exp2(fmaf(x[jj + 3], p.qscale, b4.w));
          }
        } else {
#pragma unroll
          for (int jj = 0; jj < 32; ++jj) {
            const int r = c0 + jj;
            if (t <= p.T - p.W + s_wi[r]) acc += fast_exp2(fmaf(x[jj], p.qscale, s_b[r]));
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&lempty[b]);
      for (int o = 1; o < p.pool; o <<= 1) acc += __shfl_xor_sync(kFull, acc, o);  // aligned chunks
      if (t < t_end) {
        p.s_out[(size_t)u * p.T + t] = acc;
        if (p.diag) p.diag[(size_t)u * p.T + t] = acc;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  // the MMA thread's final commit, and after an abort the copies in flight
  if (tid == 0) drain_after_abort(full, kS, abort_flag ? s_issued : 0, abort_flag ? &qfull : nullptr, &mma_done);
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tm, 512);
  }
}

// ------------------------------------------------------------ residual_tc
__global__ void __launch_bounds__(kStatsThreads, 1)
    residual_tc(const TcArgs p, const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV) {
  constexpr int kS = 2;
  extern __shared__ __align__(1024) uint8_t smraw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smraw) + 1023) & ~uintptr_t(1023));
  uint8_t* sK = sm;                        // [kS][128 x 128]
  uint8_t* sV = sm + kS * kTileBytes;      // [kS][128 x 128]
  uint8_t* sC = sm + 2 * kS * kTileBytes;  // [3 parts][128 x 128]: C0' = hi + mid + lo
  __shared__ __align__(8) uint64_t full[kS], empty[kS], yfull[2], yempty[2], mma_done;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag, s_issued;
  __shared__ float s_mv[kDP];

  const int chunk = blockIdx.x, u = blockIdx.y;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int t_begin = chunk * p.chunk;
  const int t_end = min(p.n_rows, t_begin + p.chunk);
  const int n_tiles = (max(0, t_end - t_begin) + kTok - 1) / kTok;
  volatile int* abrt = &abort_flag;
  const int D = p.D;
  const float* m0 = p.m0 + (size_t)u * rec_floats(D);

  if (tid == 0) {
    for (int i = 0; i < kS; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1 + 4);  // MMA commit + the 4 epilogue warps (value rows)
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&yfull[i], 1);
      mbar_init(&yempty[i], 4);
    }
    mbar_init(&mma_done, 1);
    abort_flag = 0;
    mbar_fence_init();
    // the first stages' copies go out while C0' is being prepared
    for (int i = kS; i < min(kS + kPF, n_tiles); ++i)
      for (int bx = 0; bx < 2; ++bx) {
        tma_prefetch_3d(&tmK, bx * 64, t_begin + i * kTok, u);
        tma_prefetch_3d(&tmV, bx * 64, t_begin + i * kTok, u);
      }
    for (int i = 0; i < min(kS, n_tiles); ++i) {
      mbar_arrive_expect_tx(&full[i], 2u * kTileBytes);
      for (int bx = 0; bx < 2; ++bx) {
        tma_load_3d(sK + i * kTileBytes + bx * kBoxBytes, &tmK, bx * 64, t_begin + i * kTok, u, &full[i]);
        tma_load_3d(sV + i * kTileBytes + bx * kBoxBytes, &tmV, bx * 64, t_begin + i * kTok, u, &full[i]);
      }
    }
    s_issued = min(kS, n_tiles);
  }
  if (warp == 1) tmem_alloc(&tmem_base, 256);
  if (warp >= 2 && warp < 6) {
    // C0' (clamped where |n0 C0| < tau) as three bf16 parts in the K-major
    // swizzled layout: row a = value dim (N), 128-byte rows over key dims (K)
    const int a = tid - 64;
    const float n0 = m0[0];
    const float tau = p.tau;
    for (int c = 0; c < kDP; c += 2) {
      float v0 = 0.f, v1 = 0.f;
      if (n0 > 0.f && a < D) {
        if (c < D) v0 = m0[4 + 2 * D + (size_t)a * D + c];
        if (c + 1 < D) v1 = m0[4 + 2 * D + (size_t)a * D + c + 1];
        if (fabsf(v0 * n0) < tau) v0 = 0.f;
        if (fabsf(v1 * n0) < tau) v1 = 0.f;
      }
      float r0 = v0, r1 = v1;
#pragma unroll
      for (int part = 0; part < 3; ++part) {
        const __nv_bfloat16 h0 = __float2bfloat16_rn(r0), h1 = __float2bfloat16_rn(r1);
        __nv_bfloat162 hv;
        hv.x = h0;
        hv.y = h1;
        *reinterpret_cast<__nv_bfloat162*>(sC + part * kTileBytes + swz_off(a, c, kTok)) = hv;
        r0 -= __bfloat162float(h0);
        r1 -= __bfloat162float(h1);
      }
    }
    s_mv[a] = (n0 > 0.f && a < D) ? m0[4 + D + a] : 0.f;
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // generic writes -> tensor-core reads
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = tmem_base;
  const float scale = rsqrtf(static_cast<float>(D));

  if (warp == 0) {
    if (lane == 0) {
      for (int i = kS; i < n_tiles; ++i) {
        const int s = i % kS, j = i / kS;
        if (kPF > 0 && i + kPF < n_tiles)
          for (int bx = 0; bx < 2; ++bx) {
            tma_prefetch_3d(&tmK, bx * 64, t_begin + (i + kPF) * kTok, u);
            tma_prefetch_3d(&tmV, bx * 64, t_begin + (i + kPF) * kTok, u);
          }
        if (!pwait(&empty[s], (j - 1) & 1, abrt, p.ws, u, p.polls)) break;
        mbar_arrive_expect_tx(&full[s], 2u * kTileBytes);
        for (int bx = 0; bx < 2; ++bx) {
          tma_load_3d(sK + s * kTileBytes + bx * kBoxBytes, &tmK, bx * 64, t_begin + i * kTok, u, &full[s]);
          tma_load_3d(sV + s * kTileBytes + bx * kBoxBytes, &tmV, bx * 64, t_begin + i * kTok, u, &full[s]);
        }
        s_issued = i + 1;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t id = idesc_bf16(128, 128, 0, 0);
      const uint32_t aC = smem_addr(sC);
      for (int i = 0; i < n_tiles; ++i) {
        const int s = i % kS, j = i / kS, b = i & 1;
        if (!pwait(&full[s], j & 1, abrt, p.ws, u, p.polls)) break;
        if (i >= 2 && !pwait(&yempty[b], ((i >> 1) - 1) & 1, abrt, p.ws, u, p.polls)) break;
        tc_fence_after();
        const uint32_t aK = smem_addr(sK + s * kTileBytes);
        for (int part = 0; part < 3; ++part)
          for (int kk = 0; kk < 8; ++kk) {
            const uint64_t dk = sdesc_sw128(aK + (kk >> 2) * kBoxBytes + (kk & 3) * 32, 16, 1024);
            const uint64_t dc =
                sdesc_sw128(aC + part * kTileBytes + (kk >> 2) * kBoxBytes + (kk & 3) * 32, 16, 1024);
            umma_bf16(tm + b * 128, dk, dc, id, (part > 0 || kk > 0) ? 1u : 0u);
          }
        umma_commit(&yfull[b]);
        umma_commit(&empty[s]);
      }
      umma_commit(&mma_done);  // every MMA issued has completed
    }
  } else {
    // two epilogue groups (warps 2..5 and 6..9) take alternate tiles; group g
    // always reads TMEM buffer g
    const int grp = (warp - 2) >> 2, qd = warp & 3;
    const uint32_t lane_base = static_cast<uint32_t>(qd * 32) << 16;
    const int row = qd * 32 + lane;  // token within the tile = TMEM lane
    for (int i = grp; i < n_tiles; i += 2) {
      const int s = i % kS, j = i / kS, b = i & 1;
      if (!pwait(&yfull[b], (i >> 1) & 1, abrt, p.ws, u, p.polls)) break;
      if (!pwait(&full[s], j & 1, abrt, p.ws, u, p.polls)) break;
      tc_fence_after();
      const uint8_t* tv = sV + s * kTileBytes;
      float ss = 0.f;
      for (int c0 = 0; c0 < kDP; c0 += 32) {
        float y[32];
        tmem_ld32(tm + lane_base + b * 128 + c0, y);
        if (c0 < D) {
#pragma unroll
          for (int jj = 0; jj < 32; jj += 8) {
            const uint4 raw = *reinterpret_cast<const uint4*>(tv + swz_off(row, c0 + jj, kTok));
            const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
              const float2 vv = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[e]));
              const int c = c0 + jj + 2 * e;
              const float r0 = vv.x - s_mv[c] - scale * y[jj + 2 * e];
              const float r1 = vv.y - s_mv[c + 1] - scale * y[jj + 2 * e + 1];
              ss = fmaf(r0, r0, fmaf(r1, r1, ss));
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        mbar_arrive(&yempty[b]);
        mbar_arrive(&empty[s]);
      }
      const int t = t_begin + i * kTok + row;
      if (t < t_end) {
        const float v =
            is_protected(t, p.T, p.W, p.sink, p.keep_window) ? 0.f : p.s_in[(size_t)u * p.T + t] * sqrtf(ss);
        p.s_out[(size_t)u * p.T + t] = v;
        if (p.diag) p.diag[(size_t)u * p.T + t] = v;
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  // the MMA thread's final commit, and after an abort the copies in flight
  if (tid == 0) drain_after_abort(full, kS, abort_flag ? s_issued : 0, nullptr, &mma_done);
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tm, 256);
  }
}

// ----------------------------------------------------------------- select
// One cluster of kSelCL CTAs per selection group -- a unit, or with the
// adaptive budget the hs KV heads of a batch item, whose (head, position)
// pairs f = h * T + t are ranked together.  R = protected + the k highest
// keys among the other pairs (ties to the lower f), written ascending, with
// each unit's count and first slot.  For one unit per group the kernel also
// gathers R's rows into dst_K/dst_V [unit][dst_cap][D] (with positions when
// the destination is a cache); a joint selection's rows are gathered by
// gather_kernel.
// Exclusive block-wide prefix sum of one int per thread; *total gets the sum.
__device__ __forceinline__ int block_excl_sum(int v, int* wsum, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(kFull, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) wsum[warp] = x;
  __syncthreads();
  if (warp == 0) {
    const int w = lane < (int)(blockDim.x >> 5) ? wsum[lane] : 0;
    int xw = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(kFull, xw, o);
      if (lane >= o) xw += y;
    }
    wsum[lane] = xw - w;
    if (lane == 31) *total = xw;
  }
  __syncthreads();
  const int r = wsum[warp] + x - v;
  __syncthreads();  // wsum is reused by the next call
  return r;
}

struct SelectArgs {
  const float* scores;  // [units][T]
  int T, W, B, sink, keep_window, D;
  const __nv_bfloat16* K;  // prompt [units][T][D]
  const __nv_bfloat16* V;
  int32_t* idx;          // [groups][hs * B] selection lists, h * T + position, ascending (workspace)
  int32_t* diag_idx;     // optional copy
  __nv_bfloat16* dst_K;  // optional (one unit per group): the rows are gathered here, [units][dst_cap][D]
  __nv_bfloat16* dst_V;
  int dst_cap;
  int32_t* dst_pos;      // optional cache bookkeeping
  int32_t* dst_len;
  int32_t* dst_seen;
  int smem_keys;  // keys of a CTA's range that the dynamic shared memory holds
  int hs;         // units per selection group (1: one unit; > 1: the KV heads of a batch item)
  const int32_t* cand;  // optional [units][Tc] ascending candidate positions per unit (null: all T)
  int Tc;               // entries per unit taking part: T, or the candidate lists' length
  int32_t* cnt;    // optional [units] rows retained per unit
  int32_t* hbeg;   // optional [units] the unit's first slot in idx
  int32_t* tile0;  // optional [groups][hs + 1] first kTok-row tile of each unit within its group, and the total
};

constexpr int kFinRB = 16;  // rows of C per finalize CTA
constexpr int kSelCL = 8;  // CTAs per selection group (one cluster), each over a contiguous range of pairs
constexpr int kSelSmemKeys = 49152;  // keys of a CTA's range cached in shared memory (192 KB)
constexpr int kMaxHs = 64;           // KV heads of a batch item with the adaptive budget

__global__ void __cluster_dims__(kSelCL, 1, 1) __launch_bounds__(kSelThreads, 2) select_kernel(const SelectArgs a) {
  __shared__ uint32_t hist[2][256];   // this CTA's histogram, double-buffered by pass parity (read remotely)
  __shared__ uint32_t whist[8][256];  // private histograms for groups of 4 warps (less atomic contention)
  __shared__ uint32_t ghist[256];     // the cluster's histogram
  __shared__ int wsum[32];
  __shared__ int tot;
  __shared__ uint32_t s_prefix;
  __shared__ int s_need;
  __shared__ int ex_cnt[2];  // this CTA's ties and certain selections (protected or above the threshold)
  __shared__ int s_before[2];
  __shared__ int s_hstart[kMaxHs + 1];  // first slot of each head in the group's selection list
  __shared__ int s_hcnt[kMaxHs];        // this CTA's selections per head (read remotely)
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = static_cast<int>(cluster.block_rank());
  const int grp = blockIdx.x / kSelCL, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int T = a.T, W = a.W, hs = a.hs;
  // entries f = h * Tc + j of the group stand for (head h, position t), t = j
  // or the candidate cand[h][j]; either way f ascending is (h, t) ascending
  const int Tc = a.Tc;
  const int N = hs * Tc;
  const int per = (N + kSelCL - 1) / kSelCL;
  const int r0 = min(N, rank * per), r1 = min(N, r0 + per);
  const float* sc = a.scores + (size_t)grp * hs * T;  // the group's units are consecutive
  const int32_t* cand = a.cand ? a.cand + (size_t)grp * N : nullptr;
  auto pos_of = [&](int f, int& h) -> int {  // (head, position) of entry f
    h = hs == 1 ? 0 : f / Tc;
    const int j = f - h * Tc;
    return cand ? cand[f] : j;
  };
  // >= 0 (validated), < candidates
  const int k = hs * (a.B - protected_count(T, W, a.sink, a.keep_window));

  // The CTA's keys are cached in shared memory when they fit (protected
  // positions hold key 0; every other position's key is at least 1, whatever
  // the bits of its score, so at most k of them are ever selected); larger
  // ranges are read from global memory on every pass.
  extern __shared__ uint32_t ks[];
  const int nk = r1 - r0;
  const bool cached = nk <= a.smem_keys;
  auto key_of = [&](int f) -> uint32_t {
    int h;
    const int t = pos_of(f, h);
    return is_protected(t, T, W, a.sink, a.keep_window) ? 0u : max(1u, float_key(sc[(size_t)h * T + t]));
  };
  auto key_at = [&](int f) -> uint32_t {  // 0 for protected positions
    return cached ? ks[f - r0] : key_of(f);
  };
  for (int h = tid; h < hs; h += kSelThreads) s_hcnt[h] = 0;
  if (cached)
    for (int i = tid; i < nk; i += kSelThreads) ks[i] = key_of(r0 + i);
  __syncthreads();
  // thread tid owns the contiguous positions [t0, t1) in the ordered passes
  const int E = (nk + kSelThreads - 1) / kSelThreads;
  const int t0 = min(r1, r0 + tid * E), t1 = min(r1, t0 + E);

  uint32_t prefix = 0, pmask = 0;
  int need = k;
  if (k > 0) {
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      for (int i = tid; i < 8 * 256; i += kSelThreads) (&whist[0][0])[i] = 0;
      __syncthreads();
      uint32_t* wh = whist[warp & 7];
#pragma unroll 4
      for (int i = tid; i < nk; i += kSelThreads) {
        const uint32_t key = key_at(r0 + i);
        if (key != 0u && (key & pmask) == prefix) atomicAdd(&wh[(key >> shift) & 255u], 1u);
      }
      __syncthreads();
      for (int i = tid; i < 256; i += kSelThreads) {
        uint32_t c = 0;
#pragma unroll
        for (int g = 0; g < 8; ++g) c += whist[g][i];
        hist[pass & 1][i] = c;
      }
      cluster.sync();  // every CTA's histogram of this pass is complete
      for (int i = tid; i < 256; i += kSelThreads) {
        uint32_t c = 0;
#pragma unroll
        for (int r = 0; r < kSelCL; ++r) c += cluster.map_shared_rank(&hist[pass & 1][0], r)[i];
        ghist[i] = c;
      }
      __syncthreads();
      if (warp == 0) {  // the digit where the descending cumulative count reaches `need`
        int cnt[8], tot8 = 0;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          cnt[e] = static_cast<int>(ghist[255 - (lane * 8 + e)]);
          tot8 += cnt[e];
        }
        int incl = tot8;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int y = __shfl_up_sync(kFull, incl, o);
          if (lane >= o) incl += y;
        }
        const int excl = incl - tot8;
        if (excl < need && incl >= need) {
          int cum = excl, e = 0;
          for (; e < 7; ++e) {
            if (cum + cnt[e] >= need) break;
            cum += cnt[e];
          }
          s_need = need - cum;
          s_prefix = prefix | (static_cast<uint32_t>(255 - (lane * 8 + e)) << shift);
        }
      }
      __syncthreads();
      need = s_need;
      prefix = s_prefix;
      pmask |= 255u << shift;
    }
  }
  // per-thread counts: protected or above the threshold key (certain), and
  // ties with it; scanned over the block, then over the cluster's ranks
  int n_tie = 0, n_sure = 0;
  for (int t = t0; t < t1; ++t) {
    const uint32_t key = key_at(t);
    if (key == 0u) {
      ++n_sure;  // protected
    } else if (k > 0) {
      n_sure += key > prefix ? 1 : 0;
      n_tie += key == prefix ? 1 : 0;
    }
  }
  const int tie_excl = block_excl_sum(n_tie, wsum, &tot);
  if (tid == 0) ex_cnt[0] = tot;
  const int sure_excl = block_excl_sum(n_sure, wsum, &tot);
  if (tid == 0) ex_cnt[1] = tot;
  (void)sure_excl;
  cluster.sync();
  if (tid == 0) {
    int ties_before = 0, sel_before = 0;
    for (int r = 0; r < rank; ++r) {
      const int* rc = cluster.map_shared_rank(ex_cnt, r);
      const int nt = rc[0], ns = rc[1];
      const int take = min(max(need - ties_before, 0), nt);  // this rank's ties that are selected
      sel_before += ns + take;
      ties_before += nt;
    }
    s_before[0] = ties_before;
    s_before[1] = sel_before;
  }
  __syncthreads();
  const int cta_ties_before = s_before[0], cta_sel_before = s_before[1];
  // this thread's selections: its certain ones and the ties that still fit
  int tb = cta_ties_before + tie_excl;
  const int my_sel = n_sure + min(max(need - tb, 0), n_tie);
  const int sel_excl = block_excl_sum(my_sel, wsum, &tot);
  const int my_first = cta_sel_before;
  int o = cta_sel_before + sel_excl;
  const int n_sel = hs * a.B;  // the group's selections (protected included)
  int32_t* out = a.idx + (size_t)grp * n_sel;
  int cur_h = 0, cur_n = 0;  // this thread's run of selections in one head (ranges rarely span two)
  for (int t = t0; t < t1; ++t) {
    const uint32_t key = key_at(t);
    bool sel = true;  // protected
    if (key != 0u) {
      const bool tie = k > 0 && key == prefix;
      sel = (k > 0 && key > prefix) || (tie && tb < need);
      tb += tie ? 1 : 0;
    }
    if (sel) {
      if (o < n_sel) {  // stored as h * T + position
        int h;
        const int pt = pos_of(t, h);
        out[o] = h * T + pt;
        if (a.diag_idx) a.diag_idx[(size_t)grp * n_sel + o] = h * T + pt;
        if (h != cur_h) {
          if (cur_n) atomicAdd(&s_hcnt[cur_h], cur_n);
          cur_h = h;
          cur_n = 0;
        }
        ++cur_n;
      }
      ++o;
    }
  }
  if (hs > 1) {
    // each head's slots are a contiguous run of the ascending list, as long
    // as the head's selections in all CTAs of the cluster
    if (cur_n) atomicAdd(&s_hcnt[cur_h], cur_n);
    cluster.sync();
    if (tid < hs) {
      int c = 0;
#pragma unroll
      for (int r = 0; r < kSelCL; ++r) c += cluster.map_shared_rank(s_hcnt, r)[tid];
      s_hstart[tid + 1] = c;
    }
    __syncthreads();
    if (tid == 0) {
      s_hstart[0] = 0;
      for (int h = 0; h < hs; ++h) s_hstart[h + 1] += s_hstart[h];
    }
  } else if (tid == 0) {
    s_hstart[0] = 0;
    s_hstart[1] = a.B;
  }
  __syncthreads();
  if (hs == 1 && a.dst_K) {
    // gather the rows this CTA selected (16-byte chunks); a joint selection's
    // rows are gathered by gather_kernel over the whole GPU instead
    const int D = a.D, per_row = D / 8, u = grp;
    const int o0 = min(my_first, n_sel), o1 = min(my_first + tot, n_sel);
    for (int i = tid; i < (o1 - o0) * per_row; i += kSelThreads) {
      const int r = o0 + i / per_row, c = i % per_row;
      const int t = min(max(out[r], 0), T - 1);  // never read outside the unit's slab
      const size_t src = ((size_t)u * T + t) * D;
      const size_t dst = ((size_t)u * a.dst_cap + r) * D;
      reinterpret_cast<uint4*>(a.dst_K + dst)[c] = reinterpret_cast<const uint4*>(a.K + src)[c];
      reinterpret_cast<uint4*>(a.dst_V + dst)[c] = reinterpret_cast<const uint4*>(a.V + src)[c];
    }
    if (a.dst_pos)
      for (int r = o0 + tid; r < o1; r += kSelThreads) a.dst_pos[(size_t)u * a.dst_cap + r] = out[r];
  }
  if (rank == 0 && tid < hs) {
    const int u = grp * hs + tid, c = s_hstart[tid + 1] - s_hstart[tid];
    if (a.cnt) a.cnt[u] = c;
    if (a.hbeg) a.hbeg[u] = grp * n_sel + s_hstart[tid];
    if (a.dst_len) {
      a.dst_len[u] = c;
      a.dst_seen[u] = T;
    }
  }
  if (rank == 0 && tid == 0 && a.tile0) {
    int acc = 0;
    for (int h = 0; h < hs; ++h) {
      a.tile0[grp * (hs + 1) + h] = acc;
      acc += (s_hstart[h + 1] - s_hstart[h] + kTok - 1) / kTok;
    }
    a.tile0[grp * (hs + 1) + hs] = acc;
  }
  cluster.sync();  // no CTA leaves while another may still read its shared memory
}

// ----------------------------------------------------------------- gather
// Copies each unit's retained rows (in list order) into dst_K/dst_V
// [unit][dst_cap][D], one kTok-row tile per CTA, with the positions when the
// destination is a cache.  With zero_pad the tile's rows past the unit's count
// are written as zeros (the moments of the slab read whole tiles).  With tile0
// the grid is (tiles of a group, groups) and each CTA finds its unit there.
struct GatherArgs {
  const int32_t* idx;    // selection lists, h * T + position
  const int32_t* hbeg;   // [units] the unit's first slot in idx
  const int32_t* cnt;    // [units] its rows
  const int32_t* tile0;  // optional [groups][hs + 1]
  int hs, T, D;
  const __nv_bfloat16* K;  // prompt [units][T][D]
  const __nv_bfloat16* V;
  __nv_bfloat16* dst_K;
  __nv_bfloat16* dst_V;
  int dst_cap;
  int32_t* dst_pos;  // optional
  int zero_pad;
};

constexpr int kGatherThreads = 512;

__global__ void __launch_bounds__(kGatherThreads) gather_kernel(const GatherArgs a) {
  int u = blockIdx.y, tile = blockIdx.x, h = 0;
  if (a.tile0) {
    const int32_t* t0 = a.tile0 + (size_t)blockIdx.y * (a.hs + 1);
    if (tile >= t0[a.hs]) return;
    while (h + 1 < a.hs && t0[h + 1] <= tile) ++h;
    u = blockIdx.y * a.hs + h;
    tile -= t0[h];
  }
  const int c = a.cnt[u];
  const int r0 = tile * kTok;
  const int r1 = min(a.zero_pad ? a.dst_cap : c, r0 + kTok);
  const int per_row = a.D / 8, per2 = 2 * per_row;  // 16-byte chunks of a row of K and V
  const int n_items = max(0, r1 - r0) * per2;
  const int32_t* lst = a.idx + a.hbeg[u];
  const int hT = h * a.T;
  constexpr int UG = 4;  // chunks in flight per thread
  for (int base = threadIdx.x; base < n_items; base += kGatherThreads * UG) {
    uint4 v[UG];
    size_t dst[UG];
    bool isV[UG];
#pragma unroll
    for (int q = 0; q < UG; ++q) {
      const int i = base + q * kGatherThreads;
      const int r = r0 + i / per2, cc = i % per2;
      isV[q] = cc >= per_row;
      const int ch = isV[q] ? cc - per_row : cc;
      dst[q] = ((size_t)u * a.dst_cap + r) * a.D + ch * 8;
      v[q] = make_uint4(0u, 0u, 0u, 0u);
      if (i < n_items && r < c) {
        const int t = min(max(lst[r] - hT, 0), a.T - 1);  // never read outside the unit's slab
        const __nv_bfloat16* src = (isV[q] ? a.V : a.K) + ((size_t)u * a.T + t) * a.D + ch * 8;
        v[q] = *reinterpret_cast<const uint4*>(src);
      }
    }
#pragma unroll
    for (int q = 0; q < UG; ++q)
      if (base + q * kGatherThreads < n_items)
        *reinterpret_cast<uint4*>((isV[q] ? a.dst_V : a.dst_K) + dst[q]) = v[q];
  }
  if (a.dst_pos)
    for (int r = r0 + threadIdx.x; r < min(c, r0 + kTok); r += kGatherThreads)
      a.dst_pos[(size_t)u * a.dst_cap + r] = lst[r] - hT;
}

// --------------------------------------------------------------- finalize
// Moments of E = all \ R for kFinRB value dims (rows of C) per CTA.  Each
// set's co-moment is the multi-way Chan merge of its chunk records, taken
// about the first chunk's means x0 so that no global mean is needed first:
//   M = sum_ch [M_ch + n_ch d_ch d_ch^T] - n dbar dbar^T,  d_ch = mu_ch - x0,
//   dbar = sum_ch n_ch d_ch / n,  mu = x0 + dbar.
// R's centred record is then removed with the reverse pairwise formula.
// merge_all = 1: the all-token set is the chunk records (its merge is kept
// in L.mall); merge_all = 0: it is L.mall itself.
//
// Thread (row ar = tid / 16, lane group cq = tid % 16) takes the columns
// cq*4 + 64h (h < D/64) of its row as float4s.  The counts and means of up to
// kFinCH records of both sets are staged in one pass; then every record's
// co-moment values are loaded with several records in flight.
constexpr int kFinCH = 32;  // records staged per pass and set
__global__ void __launch_bounds__(256) finalize_kernel(const Layout L, float* out_rec, mkv_moments out_mom,
                                                       int final_out, int merge_all) {
  constexpr int RB = kFinRB, NV = kDP / 64;  // NV float4s per thread (D = 128; one at D = 64)
  __shared__ float s_n[2][kFinCH];
  __shared__ __align__(16) float s_mv[2][kFinCH][RB];
  __shared__ __align__(16) float s_mk[2][kFinCH][kDP];
  const int D = L.D;
  const int nv = D / 64;
  const int rb = blockIdx.x, u = blockIdx.y, tid = threadIdx.x;
  const size_t rf = rec_floats(D);
  const int ar = tid / 16, cq = tid % 16;
  const int row = rb * RB + ar;

  const int n_rec = merge_all ? L.n_chunks : 1;
  const float* recA = merge_all ? L.mpart + (size_t)u * L.n_chunks * rf : L.mall + (size_t)u * rf;
  const float* recR = L.rpart + (size_t)u * L.n_rchunks * rf;
  // a joint selection leaves the unit's rows in its first ceil(cnt / kTok) records
  const int n_rrec = L.hs > 1 ? min(L.n_rchunks, (L.cnt[u] + kTok - 1) / kTok) : L.n_rchunks;

  struct Set {
    float n, sv, sk[4 * NV], M[4 * NV];
    float x0v, x0k[4 * NV];
  };
  Set A{}, R{};
  auto merge = [&](Set& st, int set, const float* rbase, int g0, int nb) {
#pragma unroll 4
    for (int ch = 0; ch < nb; ++ch) {
      const float* m = rbase + (size_t)(g0 + ch) * rf + 4 + 2 * D + (size_t)row * D;
      float4 mv4[NV];
#pragma unroll
      for (int h = 0; h < NV; ++h)
        mv4[h] = h < nv ? *reinterpret_cast<const float4*>(m + h * 64 + cq * 4) : make_float4(0.f, 0.f, 0.f, 0.f);
      const float nc = s_n[set][ch];
      if (nc > 0.f) {  // an empty record's co-moment is never written
        const float dv = s_mv[set][ch][ar] - st.x0v;
        st.n += nc;
        st.sv = fmaf(nc, dv, st.sv);
#pragma unroll
        for (int h = 0; h < NV; ++h) {
          if (h >= nv) break;
          const float4 k4 = *reinterpret_cast<const float4*>(&s_mk[set][ch][h * 64 + cq * 4]);
          const float kk[4] = {k4.x, k4.y, k4.z, k4.w}, mm[4] = {mv4[h].x, mv4[h].y, mv4[h].z, mv4[h].w};
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const float dk = kk[i] - st.x0k[h * 4 + i];
            st.sk[h * 4 + i] = fmaf(nc, dk, st.sk[h * 4 + i]);
            st.M[h * 4 + i] += mm[i] + nc * dv * dk;
          }
        }
      }
    }
  };
  for (int g0 = 0; g0 < max(n_rec, n_rrec); g0 += kFinCH) {
    const int nbA = max(0, min(kFinCH, n_rec - g0)), nbR = max(0, min(kFinCH, n_rrec - g0));
    if (g0 > 0) __syncthreads();
    // per record: (n, ...), the CTA's RB mu_v rows and mu_k as float4s;
    // four loads per thread in flight before their stores
    const int per = 1 + RB / 4 + D / 4, totA = nbA * per, tot = totA + nbR * per;
    for (int i0 = 0; i0 < tot; i0 += 4 * 256) {
      float4 v[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int i = i0 + k * 256 + tid;
        if (i < tot) {
          const int set = i >= totA, kk = set ? i - totA : i, ch = kk / per, j = kk % per;
          const float* r = (set ? recR : recA) + (size_t)(g0 + ch) * rf;
          const float* src = j == 0 ? r : (j <= RB / 4 ? r + 4 + D + rb * RB + (j - 1) * 4 : r + 4 + (j - 1 - RB / 4) * 4);
          v[k] = *reinterpret_cast<const float4*>(src);
        }
      }
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const int i = i0 + k * 256 + tid;
        if (i < tot) {
          const int set = i >= totA, kk = set ? i - totA : i, ch = kk / per, j = kk % per;
          if (j == 0) s_n[set][ch] = v[k].x;
          else if (j <= RB / 4) *reinterpret_cast<float4*>(&s_mv[set][ch][(j - 1) * 4]) = v[k];
          else *reinterpret_cast<float4*>(&s_mk[set][ch][(j - 1 - RB / 4) * 4]) = v[k];
        }
      }
    }
    __syncthreads();
    if (g0 == 0) {  // the first record's means (zero when a set has none)
      A.x0v = nbA > 0 ? s_mv[0][0][ar] : 0.f;
      R.x0v = nbR > 0 ? s_mv[1][0][ar] : 0.f;
#pragma unroll
      for (int h = 0; h < NV; ++h)
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int c = h * 64 + cq * 4 + i;
          A.x0k[h * 4 + i] = (nbA > 0 && h < nv) ? s_mk[0][0][c] : 0.f;
          R.x0k[h * 4 + i] = (nbR > 0 && h < nv) ? s_mk[1][0][c] : 0.f;
        }
    }
    merge(A, 0, recA, g0, nbA);
    merge(R, 1, recR, g0, nbR);
  }

  const float n = A.n, nR = R.n, nE = n - nR;
  const float mv = A.x0v + A.sv / n;
  const float mvR = nR > 0.f ? R.x0v + R.sv / nR : 0.f;
  const float mvE = nE > 0.f ? (n * mv - nR * mvR) / nE : 0.f;
  float* mall = L.mall + (size_t)u * rf;
  float* o = final_out ? nullptr : out_rec + (size_t)u * rf;
#pragma unroll
  for (int h = 0; h < NV; ++h) {
    if (h >= nv) break;
    float Mo[4], CE[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int j = h * 4 + i, c = h * 64 + cq * 4 + i;
      const float mk = A.x0k[j] + A.sk[j] / n;
      const float M = A.M[j] - A.sv * A.sk[j] / n;
      const float mkR = nR > 0.f ? R.x0k[j] + R.sk[j] / nR : 0.f;
      const float MR = nR > 0.f ? R.M[j] - R.sv * R.sk[j] / nR : 0.f;
      Mo[i] = M;
      CE[i] = 0.f;
      float mkE = 0.f;
      if (nE > 0.f) {
        mkE = (n * mk - nR * mkR) / nE;
        const float ME = M - MR - (nE * nR / n) * (mvR - mvE) * (mkR - mkE);
        CE[i] = ME / nE;
      }
      if (rb == 0 && ar == 0) {  // the k means: row 0's threads
        if (merge_all) mall[4 + c] = mk;
        if (final_out) out_mom.mu_k[(size_t)u * D + c] = mkE;
        else o[4 + c] = mkE;
      }
    }
    const size_t e = (size_t)row * D + h * 64 + cq * 4;
    if (merge_all) *reinterpret_cast<float4*>(mall + 4 + 2 * D + e) = make_float4(Mo[0], Mo[1], Mo[2], Mo[3]);
    if (final_out) *reinterpret_cast<float4*>(out_mom.C + (size_t)u * D * D + e) = make_float4(CE[0], CE[1], CE[2], CE[3]);
    else *reinterpret_cast<float4*>(o + 4 + 2 * D + e) = make_float4(CE[0], CE[1], CE[2], CE[3]);
  }
  if (cq == 0) {  // the v means: one thread per row
    if (merge_all) mall[4 + D + row] = mv;
    if (final_out) out_mom.mu_v[(size_t)u * D + row] = mvE;
    else o[4 + D + row] = mvE;
  }
  if (rb == 0 && tid == 0) {
    if (merge_all) mall[0] = n;
    if (final_out) out_mom.n[u] = static_cast<int32_t>(nE);
    else o[0] = nE;
  }
}

// ---------------------------------------------------------- keep-all path
template <int D>
__global__ void __launch_bounds__(256) keep_all_kernel(const CompressArgs a, int T) {
  const int u = blockIdx.y;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = blockIdx.x * 8 + warp;
  if (i < T) {
    const __nv_bfloat16* Ks = reinterpret_cast<const __nv_bfloat16*>(a.K) + ((size_t)u * T + i) * D;
    const __nv_bfloat16* Vs = reinterpret_cast<const __nv_bfloat16*>(a.V) + ((size_t)u * T + i) * D;
    __nv_bfloat16* Kd = reinterpret_cast<__nv_bfloat16*>(a.cache.K) + ((size_t)u * a.cache.capacity + i) * D;
    __nv_bfloat16* Vd = reinterpret_cast<__nv_bfloat16*>(a.cache.V) + ((size_t)u * a.cache.capacity + i) * D;
    for (int c = lane * 2; c < D; c += 64) {
      *reinterpret_cast<__nv_bfloat162*>(Kd + c) = *reinterpret_cast<const __nv_bfloat162*>(Ks + c);
      *reinterpret_cast<__nv_bfloat162*>(Vd + c) = *reinterpret_cast<const __nv_bfloat162*>(Vs + c);
    }
    if (lane == 0) a.cache.pos[(size_t)u * a.cache.capacity + i] = i;
  }
  if (blockIdx.x == 0) {
    if (threadIdx.x == 0) {
      a.cache.len[u] = T;
      a.cache.seen[u] = T;
      a.mom.n[u] = 0;
    }
    for (int e = threadIdx.x; e < D * D; e += blockDim.x) a.mom.C[(size_t)u * D * D + e] = 0.f;
    for (int e = threadIdx.x; e < D; e += blockDim.x) {
      a.mom.mu_k[(size_t)u * D + e] = 0.f;
      a.mom.mu_v[(size_t)u * D + e] = 0.f;
    }
  }
}

// ------------------------------------------------------------------- host
constexpr size_t kStatsSmem = 1024 + 2 * 2 * kTileBytes + 2 * 2 * kBoxBytes + 4096;  // K, V stages, Q, ones
constexpr size_t kStats0Smem = 1024 + 2 * kTileBytes + 4096;                            // one K, V stage, ones
constexpr size_t kScoresSmem = 1024 + 3 * kTileBytes + 2 * 2 * kBoxBytes;
constexpr size_t kResidualSmem = 1024 + 2 * 2 * kTileBytes + 3 * kTileBytes;

cudaError_t run(const CompressArgs& a, const mkv_geom& g, int num_sms, cudaStream_t st) {
  Layout L = make_layout(g, a.T, a.budget, a.window, a.sink, a.keep_window, a.adaptive, num_sms);
  carve(L, a.ws);
  const int D = g.head_dim, T = a.T, B = a.budget, U = L.units, Bc = L.Bcap;
  const bool joint = L.hs > 1;
  const bool keep_all = T <= B;
  cudaError_t e = cudaSuccess;
  auto attr = [](const void* f, size_t bytes) {
    return cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes));
  };
  if ((e = attr((const void*)stats_tc<1>, kStatsSmem)) != cudaSuccess) return e;
  if ((e = attr((const void*)stats_tc<0>, kStats0Smem)) != cudaSuccess) return e;
  if ((e = attr((const void*)scores_tc, kScoresSmem)) != cudaSuccess) return e;
  if ((e = attr((const void*)residual_tc, kResidualSmem)) != cudaSuccess) return e;

  CUtensorMap tmK, tmV, tmQ, tmGK, tmGV, tmCK, tmCV;
  const uint64_t rs = (uint64_t)D * 2;
  bool ok = encode_tmap_bf16_3d(&tmK, a.K, D, T, U, rs, (uint64_t)T * rs, kTok) &&
            encode_tmap_bf16_3d(&tmV, a.V, D, T, U, rs, (uint64_t)T * rs, kTok) &&
            encode_tmap_bf16_3d(&tmQ, a.Q, D, L.RW, U, rs, (uint64_t)L.RW * rs, L.RWb * 128);
  // the retained rows: B per unit, or (joint) up to the capacity with the
  // rows past each unit's count zero up to the tile (or outside the map)
  const int cache_rows = joint ? a.cache.capacity : B;
  if (!keep_all)
    ok = ok && encode_tmap_bf16_3d(&tmGK, L.gK, D, Bc, U, rs, (uint64_t)Bc * rs, kTok) &&
         encode_tmap_bf16_3d(&tmGV, L.gV, D, Bc, U, rs, (uint64_t)Bc * rs, kTok) &&
         encode_tmap_bf16_3d(&tmCK, a.cache.K, D, cache_rows, U, rs, (uint64_t)a.cache.capacity * rs, kTok) &&
         encode_tmap_bf16_3d(&tmCV, a.cache.V, D, cache_rows, U, rs, (uint64_t)a.cache.capacity * rs, kTok);
  if (!ok) return cudaErrorInvalidValue;

  TcArgs tp{};
  tp.D = D;
  tp.RW = L.RW;
  tp.RWb = L.RWb;
  tp.W = a.window;
  tp.T = T;
  tp.causal = a.causal;
  tp.sink = a.sink;
  tp.keep_window = a.keep_window;
  tp.pool = a.pool;
  tp.qscale = rsqrtf(static_cast<float>(D)) * kLog2e;
  tp.tau = a.tau;
  tp.ws = a.ws;
  tp.polls = pipeline_poll_limit();
  const dim3 cg(L.n_chunks, U);

  if (!keep_all || a.diag_scores != nullptr) {
    TcArgs p1 = tp;
    p1.n_rows = T;
    p1.chunk = L.chunk;
    p1.n_chunks = L.n_chunks;
    p1.rowpart = L.rowpart;
    p1.mrec = L.mpart;
    stats_tc<1><<<cg, kStatsThreads, kStatsSmem, st>>>(p1, tmK, tmV, tmQ);
    TcArgs p2 = p1;
    p2.s_out = L.s;
    p2.diag = a.diag_scores;
    scores_tc<<<cg, kStatsThreads, kScoresSmem, st>>>(p2, tmK, tmQ);
  }
  if (keep_all) {
    if (D == 128) keep_all_kernel<128><<<dim3((T + 7) / 8, U), 256, 0, st>>>(a, T);
    else keep_all_kernel<64><<<dim3((T + 7) / 8, U), 256, 0, st>>>(a, T);
    return cudaGetLastError();
  }

  SelectArgs sa{};
  const int n_groups = U / L.hs;
  const bool prefilter = L.cand != nullptr;
  // keys a CTA caches when its range fits, for the joint (or per-unit) selection and the prefilter
  auto cached_keys = [](long per) { return per <= kSelSmemKeys ? static_cast<int>(per) : 0; };
  sa.smem_keys = cached_keys((L.hs * (long)L.Tc + kSelCL - 1) / kSelCL);
  const int pf_keys = cached_keys((T + kSelCL - 1) / kSelCL);
  const size_t sel_smem = (size_t)sa.smem_keys * sizeof(uint32_t), pf_smem = (size_t)pf_keys * sizeof(uint32_t);
  if ((e = attr((const void*)select_kernel, std::max(sel_smem, pf_smem))) != cudaSuccess) return e;
  sa.T = T;
  sa.Tc = L.Tc;
  sa.cand = L.cand;
  sa.W = a.window;
  sa.B = B;
  sa.sink = a.sink;
  sa.keep_window = a.keep_window;
  sa.D = D;
  sa.K = static_cast<const __nv_bfloat16*>(a.K);
  sa.V = static_cast<const __nv_bfloat16*>(a.V);
  sa.idx = L.idx;
  sa.hs = L.hs;
  sa.cnt = L.cnt;
  sa.hbeg = L.hbeg;
  sa.tile0 = joint ? L.tile0 : nullptr;
  // the candidates of a joint selection over `scores`: each unit's protected
  // rows and its top Tc - |protected| (a per-unit selection)
  auto prefilter_launch = [&](const float* scores) {
    if (!prefilter) return;
    SelectArgs pf = sa;
    pf.scores = scores;
    pf.hs = 1;
    pf.Tc = T;
    pf.cand = nullptr;
    pf.B = L.Tc;
    pf.idx = L.cand;
    pf.smem_keys = pf_keys;
    pf.cnt = nullptr;
    pf.hbeg = nullptr;
    pf.tile0 = nullptr;
    select_kernel<<<U * kSelCL, kSelThreads, pf_smem, st>>>(pf);
  };
  // the retained rows' tiles: (chunks, units), or (a group's tiles, groups)
  const dim3 tiles = joint ? dim3(L.gtiles, n_groups) : dim3(L.n_rchunks, U);
  GatherArgs ga{};
  ga.idx = L.idx;
  ga.hbeg = L.hbeg;
  ga.cnt = L.cnt;
  ga.tile0 = sa.tile0;
  ga.hs = L.hs;
  ga.T = T;
  ga.D = D;
  ga.K = sa.K;
  ga.V = sa.V;
  ga.zero_pad = joint ? 1 : 0;
  TcArgs rset = tp;  // moments of a dense row set: chunks of kTok rows
  rset.n_rows = Bc;
  rset.rows_u = joint ? L.cnt : nullptr;
  rset.tile0 = sa.tile0;
  rset.hs = L.hs;
  rset.chunk = kTok;
  rset.n_chunks = L.n_rchunks;
  rset.mrec = L.rpart;

  if (a.mi) {
    SelectArgs s0 = sa;
    s0.scores = L.s;
    s0.diag_idx = a.diag_idx1;
    GatherArgs g0 = ga;
    g0.dst_K = L.gK;
    g0.dst_V = L.gV;
    g0.dst_cap = Bc;
    if (!joint) {
      s0.dst_K = g0.dst_K;
      s0.dst_V = g0.dst_V;
      s0.dst_cap = g0.dst_cap;
    }
    prefilter_launch(L.s);
    select_kernel<<<n_groups * kSelCL, kSelThreads, sel_smem, st>>>(s0);
    if (joint) gather_kernel<<<tiles, kGatherThreads, 0, st>>>(g0);
    stats_tc<0><<<tiles, kStatsThreads, kStats0Smem, st>>>(rset, tmGK, tmGV, tmQ);
    finalize_kernel<<<dim3(D / kFinRB, U), 256, 0, st>>>(L, L.m0, a.mom, 0, 1);
    TcArgs r = tp;
    r.n_rows = T;
    r.chunk = L.chunk;
    r.n_chunks = L.n_chunks;
    r.m0 = L.m0;
    r.s_in = L.s;
    r.s_out = L.s2;
    r.diag = a.diag_score2;
    residual_tc<<<cg, kStatsThreads, kResidualSmem, st>>>(r, tmK, tmV);
  }
  SelectArgs s1 = sa;
  s1.scores = a.mi ? L.s2 : L.s;
  s1.diag_idx = a.mi ? nullptr : a.diag_idx1;
  s1.dst_len = a.cache.len;
  s1.dst_seen = a.cache.seen;
  GatherArgs g1 = ga;
  g1.dst_K = static_cast<__nv_bfloat16*>(a.cache.K);
  g1.dst_V = static_cast<__nv_bfloat16*>(a.cache.V);
  g1.dst_cap = a.cache.capacity;
  g1.dst_pos = a.cache.pos;
  if (!joint) {
    s1.dst_K = g1.dst_K;
    s1.dst_V = g1.dst_V;
    s1.dst_cap = g1.dst_cap;
    s1.dst_pos = g1.dst_pos;
  }
  prefilter_launch(s1.scores);
  select_kernel<<<n_groups * kSelCL, kSelThreads, sel_smem, st>>>(s1);
  if (joint) gather_kernel<<<tiles, kGatherThreads, 0, st>>>(g1);
  stats_tc<0><<<tiles, kStatsThreads, kStats0Smem, st>>>(rset, tmCK, tmCV, tmQ);
  finalize_kernel<<<dim3(D / kFinRB, U), 256, 0, st>>>(L, nullptr, a.mom, 1, a.mi ? 0 : 1);
  return cudaGetLastError();
}

}  // namespace

size_t compress_workspace_bytes(const mkv_geom& g, int32_t T, const mkv_compress_params& p, int num_sms) {
  Layout L = make_layout(g, T, p.budget, p.window, p.sink, p.keep_window, p.adaptive, num_sms);
  return carve(L, nullptr);
}

cudaError_t launch_compress(const CompressArgs& a, const mkv_geom& g, size_t ws_bytes, int num_sms,
                            cudaStream_t stream) {
  (void)ws_bytes;
  if (g.head_dim != 128 && g.head_dim != 64) return cudaErrorInvalidValue;
  return run(a, g, num_sms, stream);
}

}  // namespace mkv
