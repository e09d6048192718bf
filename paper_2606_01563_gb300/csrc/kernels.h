// Internal launcher interface between the C-ABI layer (api.cu) and the kernels.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/mkv.h"

namespace mkv {

// ------------------------------------------------------------------ decode
struct DecodeArgs {
  const void* q;      // bf16 [b, Hkv*G, D]
  const void* k_new;  // bf16 [b, Hkv, D] or null
  const void* v_new;
  void* K;            // bf16 [b, Hkv, cap, D]
  void* V;
  int32_t* pos;
  int32_t* len;
  int32_t* seen;
  int32_t cap;
  const int32_t* n;
  const float* mu_k;
  const float* mu_v;
  const float* C;
  const __nv_bfloat16* C16;  // optional bf16 copy of C (read instead of C when set)
  const uint2* Cs;           // optional operand form of C' (bf16x2 hi, lo words per column pair; read instead of C)
  int32_t correction;
  int32_t order;
  float tau;
  float* out;
  float* lse;
  void* ws;            // workspace header (error word)
  uint32_t* counters;  // [units]
  float* partial;      // [units][S][G][D+4]
  float* fhat;         // [units][G][D]
  int32_t batch;
  int32_t n_kv;
  int32_t S;       // split count of the ticket kernel (its partial records are sized for it)
  int32_t S_cl;    // split count of the cluster kernel; 0 when no cluster of that size fits
  uint32_t polls;  // poll limit of the tile waits (the drain after a timeout uses kMaxPolls)
  int32_t early;   // cache and moments read before the dependency wait (mkv_decode_params.early_load)
};

constexpr int kDecodeTile = 64;  // tokens per pipeline stage

int decode_splits(const mkv_geom& g, int32_t capacity, int num_sms);
int decode_cluster_splits(const mkv_geom& g, int32_t capacity, int num_sms, int early);
size_t decode_workspace_bytes(const mkv_geom& g, int32_t capacity, int num_sms);
// Carves the workspace and fills the ws/counters/partial/fhat fields.
void decode_carve(DecodeArgs& a, const mkv_geom& g, int32_t capacity, int num_sms, void* ws);
// The cluster kernel when a.S_cl > 0 (and the ticket merge is not forced), else the ticket kernel.
cudaError_t launch_decode(const DecodeArgs& a, int head_dim, int group, cudaStream_t stream);
cudaError_t launch_decode_cluster(const DecodeArgs& a, int head_dim, int group, cudaStream_t stream);
cudaError_t launch_pack_bf16(const float* C, __nv_bfloat16* C16, size_t n, cudaStream_t stream);
cudaError_t launch_pack_split(const float* C, const int32_t* n, float tau, uint2* Cs, int units, int D,
                              cudaStream_t stream);

// ------------------------------------------------------------------- evict
struct EvictArgs {
  const void* q;      // bf16 [b, Hkv*G, D]
  const void* k_new;  // bf16 [b, Hkv, D] or null
  const void* v_new;
  void* K;
  void* V;
  int32_t* pos;
  int32_t* len;
  int32_t* seen;
  int32_t cap;
  int32_t* n;
  float* mu_k;
  float* mu_v;
  float* C;
  int32_t budget;
  float tau;
  void* ws;
  float* scratch;  // [units][G][cap] logits (single-CTA kernel)
  void* stage;     // [units][cap] rows staged by the cluster kernel's compaction
  float* Y;          // optional fp32 [units][cap][D]: y_j = S_tilde k_j of each row (mkv_cache.y)
  int32_t* y_len;    // optional [units]: rows 0..y_len-1 of Y are current (mkv_cache.y_len)
  int32_t rows_max;  // cluster kernel: rows per CTA slice = ceil(cap / CTAs per unit)
  int32_t kv_smem;   // cluster kernel: the slice's K/V rows are cached in shared memory
  int32_t batch;
  int32_t n_kv;
};

size_t evict_workspace_bytes(const mkv_geom& g, int32_t capacity);
void evict_carve(EvictArgs& a, const mkv_geom& g, int32_t capacity, void* ws);
cudaError_t launch_evict(const EvictArgs& a, int head_dim, int group, cudaStream_t stream);

// ---------------------------------------------------------------- compress
struct CompressArgs {
  const void* K;      // bf16 [b, Hkv, T, D]
  const void* V;
  const void* Q;      // bf16 [b, Hkv, G, w, D]
  int32_t T;
  int32_t budget;
  int32_t window;
  int32_t sink;
  int32_t keep_window;
  int32_t pool;
  int32_t mi;
  int32_t causal;
  float tau;
  int32_t adaptive;   // 1: joint selection over the KV heads of each batch item
  mkv_cache cache;
  mkv_moments mom;
  float* diag_scores;
  float* diag_score2;
  int32_t* diag_idx1;
  void* ws;
  int32_t batch;
  int32_t n_kv;
};

size_t compress_workspace_bytes(const mkv_geom& g, int32_t T, const mkv_compress_params& p,
                                int num_sms);
cudaError_t launch_compress(const CompressArgs& a, const mkv_geom& g, size_t ws_bytes, int num_sms,
                            cudaStream_t stream);

}  // namespace mkv
