// Host-side helpers shared by the C-ABI entry points: the argument checks
// (so that every entry point that launches a given kernel rejects exactly the
// same inputs) and an NVTX range per call.
#pragma once

#include <nvtx3/nvToolsExt.h>
#include <stdint.h>

#include "../../include/mkv.h"

namespace mkv {

// An NVTX range named after the entry point, open for the call's host-side
// duration (argument checks and launches): a profiler's timeline shows which
// call launched which kernels.  Without a profiler attached it costs a branch.
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
};

inline bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// batch and KV heads are grid dimensions of the decode launch (z and y), so
// each stays within 65535
inline bool geom_ok(const mkv_geom& g) {
  return g.batch >= 1 && g.n_kv_heads >= 1 && g.batch <= 65535 && g.n_kv_heads <= 65535 &&
         (g.head_dim == 64 || g.head_dim == 128) && (g.group == 1 || g.group == 2 || g.group == 4 || g.group == 8) &&
         (long)g.batch * g.n_kv_heads <= 65535L * 64;
}

// status for a geometry geom_ok rejects: an unbuilt head_dim is unsupported,
// anything else is a shape error
inline mkv_status geom_status(const mkv_geom& g) {
  return (g.head_dim == 64 || g.head_dim == 128) ? MKV_ERR_SHAPE : MKV_ERR_UNSUPPORTED;
}

// K and V rows are read by 16-byte tensor copies; the optional y rows by
// vector loads, and y comes with y_len or not at all
inline bool cache_ok(const mkv_cache* c) {
  return c && c->K && c->V && c->pos && c->len && c->seen && c->capacity >= 1 && aligned(c->K, 16) &&
         aligned(c->V, 16) && ((c->y == nullptr) == (c->y_len == nullptr)) && aligned(c->y, 16);
}

// The decode kernel reads mu_k as float2 and mu_v (and C) as float4, so mu_k
// must be 8-byte and mu_v and C 16-byte aligned; a misaligned vector load
// would fault on the device instead of failing here.
inline bool moments_ok(const mkv_moments* m) {
  return m && m->n && m->mu_k && m->mu_v && m->C && aligned(m->C, 16) && aligned(m->mu_k, 8) &&
         aligned(m->mu_v, 16);
}

// Every check of a decode step except the workspace (Algorithm 1 Phase 2
// inputs): MKV_OK or the status the entry point returns.
inline mkv_status decode_args_status(const mkv_geom& geom, const void* q, const void* k_new, const void* v_new,
                                     const mkv_cache* cache, const mkv_moments* mom, const mkv_decode_params* p,
                                     const float* out) {
  if (!geom_ok(geom)) return geom_status(geom);
  if (!q || !out || !p || !cache_ok(cache)) return MKV_ERR_INVALID_ARG;
  if ((k_new == nullptr) != (v_new == nullptr)) return MKV_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(out, 16) || (k_new && (!aligned(k_new, 16) || !aligned(v_new, 16))))
    return MKV_ERR_INVALID_ARG;
  if (p->correction != 0 && p->correction != 1) return MKV_ERR_INVALID_ARG;
  if (p->order != 0 && p->order != 1) return MKV_ERR_INVALID_ARG;
  if (p->correction && !moments_ok(mom)) return MKV_ERR_INVALID_ARG;
  if (!(p->tau >= 0.f)) return MKV_ERR_INVALID_ARG;
  if (p->C16 && !aligned(p->C16, 16)) return MKV_ERR_INVALID_ARG;
  if (p->C_split && (!aligned(p->C_split, 16) || p->C16)) return MKV_ERR_INVALID_ARG;
  if (p->early_load != 0 && p->early_load != 1) return MKV_ERR_INVALID_ARG;
  return MKV_OK;
}

}  // namespace mkv
