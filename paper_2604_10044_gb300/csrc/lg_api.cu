// C ABI of liblg.so (include/lg.h): host-side validation, workspace layout and launches.
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <string.h>

#include "lg.h"
#include "lg_internal.h"

namespace {

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

lg_status check_cache(const lg_cache *c) {
  if (!c || !c->k || !c->v || !c->seq_off || !c->cap || !c->len || !c->dev_status)
    return LG_ERR_INVALID_ARG;
  if (!aligned16(c->k) || !aligned16(c->v) || !aligned16(c->sketch)) return LG_ERR_INVALID_ARG;
  if (c->dtype != LG_BF16 && c->dtype != LG_F32) return LG_ERR_UNSUPPORTED;
  if (c->d != 64 && c->d != 128) return LG_ERR_UNSUPPORTED;
  if (c->L < 1 || c->H_kv < 1 || c->batch < 1 || c->S_total < 1) return LG_ERR_INVALID_ARG;
  if ((c->H_kv * c->d) % 128) return LG_ERR_UNSUPPORTED;  // sketch rows of whole 16-byte chunks
  if ((c->h2o == nullptr) != (c->pos == nullptr)) return LG_ERR_INVALID_ARG;
  return LG_OK;
}

lg_status check_params(const lg_guard_params *p) {
  if (!p) return LG_ERR_INVALID_ARG;
  if (p->W < 1 || p->K < 0 || p->K > 3 || p->n_anchor < 0 || p->stall_len < 0 || p->p_min < 1 ||
      p->p_max < p->p_min || p->m_rep < 1 || p->l_min < 0 || p->suffix_w < 1 ||
      p->level_max < 0 || p->level_max > 30 || p->headroom < 0 || p->cooldown < 0)
    return LG_ERR_INVALID_ARG;
  if (!(p->tau_ham >= 0.0 && p->tau_ham <= 1.0)) return LG_ERR_INVALID_ARG;
  return LG_OK;
}

lg_status cuda_status(cudaError_t e) { return e == cudaSuccess ? LG_OK : LG_ERR_CUDA; }

// the token monitor's history must hold the window and every period test's reads
lg_status check_token_params(const lg_guard_params *p, const lg_token_params *tp) {
  if (!tp) return LG_ERR_INVALID_ARG;
  if (tp->cr_every < 1 || tp->theta_streak < 0 || !(tp->theta_cr >= 0.0) ||
      !(tp->theta_conf >= 0.0))
    return LG_ERR_INVALID_ARG;
  const int64_t tail = p->m_rep * (int64_t)p->p_max > p->l_min ? p->m_rep * (int64_t)p->p_max
                                                               : (int64_t)p->l_min;
  if (tp->hist < p->W || tp->hist < p->p_max + tail || tp->hist > 8192 || p->W > 4096)
    return LG_ERR_UNSUPPORTED;
  return LG_OK;
}

// rows per chunk of the fp32 path (one work item: one CTA), a multiple of the staging tile,
// twelve CTAs per SM of a 152-SM GB300, at most 2048 rows; for the bf16 path it only sizes the
// workspace (the kernel picks its own chunk rows from the call's lengths, never more chunks
// per group than the workspace holds): about eight chunks per SM, at most 4096 rows
int attend_chunk_rows(const lg_cache *c, int n_layers, int max_len) {
  const int tile = lg::attend_tile_rows(c->dtype, c->d);
  const int64_t rows = (int64_t)max_len * c->batch * c->H_kv * n_layers;
  const int64_t target = c->dtype == LG_BF16 ? 152 * 8 : 152 * 3 * 4;
  int64_t ch = (rows + target - 1) / target;
  ch = (ch + tile - 1) / tile * tile;
  const int64_t lo = c->dtype == LG_BF16 ? tile : 2 * tile;
  const int64_t hi = c->dtype == LG_BF16 ? 4096 : 2048 / tile * tile;
  if (ch < lo) ch = lo;
  if (ch > hi) ch = hi;
  return (int)ch;
}

struct AttendLayout {
  int chunk_rows, max_chunks;
  size_t partial_bytes, final_bytes, logits_bytes, counter_bytes, total;
};

size_t round256(size_t x) { return (x + 255) / 256 * 256; }

AttendLayout attend_layout(const lg_cache *c, int H_q, int n_layers, int max_len, int h2o) {
  AttendLayout L;
  L.chunk_rows = attend_chunk_rows(c, n_layers, max_len);
  L.max_chunks = (max_len + L.chunk_rows - 1) / L.chunk_rows;
  if (L.max_chunks < 1) L.max_chunks = 1;
  L.partial_bytes =
      round256((size_t)n_layers * c->batch * H_q * L.max_chunks * (c->d + 8) * sizeof(float));
  L.final_bytes = h2o ? round256((size_t)n_layers * c->batch * H_q * 2 * sizeof(float)) : 0;
  L.logits_bytes =
      h2o ? round256((size_t)n_layers * c->H_kv * c->S_total * (H_q / c->H_kv) * sizeof(float))
          : 0;
  // chunk counter, one arrival counter per group, and the pass-direction word
  L.counter_bytes = round256((size_t)(2 + (int64_t)n_layers * c->batch * c->H_kv) * sizeof(int));
  L.total = L.partial_bytes + L.final_bytes + L.logits_bytes + L.counter_bytes;
  return L;
}

}  // namespace

extern "C" {

lg_status lg_default_params(lg_guard_params *p) {
  if (!p) return LG_ERR_INVALID_ARG;
  memset(p, 0, sizeof(*p));
  p->W = 256;          // Sec. 6.1
  p->K = 2;            // Sec. 6.1
  p->t_min = 64;       // App. B.2
  p->cooldown = 32;    // App. B.2
  p->n_anchor = 32;    // Sec. 6.1
  p->stall_len = 4;    // App. B.2
  p->p_min = 1;
  p->p_max = 128;
  p->l_min = 32;
  p->m_rep = 3;
  p->suffix_w = 64;
  p->guard_layer = 0;
  p->level_max = 3;
  p->retrig_window = 64;
  p->headroom = 64;
  p->theta_ttr = 0.2;  // App. B.2
  p->theta_nov = 0.02; // App. B.2
  p->theta_ent = 0.7;
  p->theta_lift = 2.0;
  p->tau_ham = 0.125;
  return LG_OK;
}

const char *lg_status_string(lg_status s) {
  switch (s) {
    case LG_OK: return "ok";
    case LG_ERR_INVALID_ARG: return "invalid argument";
    case LG_ERR_UNSUPPORTED: return "unsupported shape or dtype";
    case LG_ERR_CUDA: return "CUDA launch failed";
    case LG_ERR_CAPACITY: return "sequence length above its capacity or max_len";
    case LG_ERR_TIMEOUT: return "bounded wait ran out";
    case LG_ERR_WORKSPACE: return "workspace missing or too small";
    case LG_ERR_BUDGET: return "budget too small for the retained set";
  }
  return "unknown status";
}

size_t lg_workspace_size(const lg_cache *c, int H_q, int n_layers, int max_len,
                         int accumulate_h2o) {
  if (check_cache(c) != LG_OK || H_q < 1 || n_layers < 1 || max_len < 1) return 0;
  return attend_layout(c, H_q, n_layers, max_len, accumulate_h2o).total;
}

lg_status lg_state_init(const lg_cache *c, lg_guard_state *state, int t_gen0, cudaStream_t s) {
  lg_status st = check_cache(c);
  if (st != LG_OK) return st;
  if (!state) return LG_ERR_INVALID_ARG;
  return cuda_status(lg::launch_state_init(*c, state, t_gen0, s));
}

lg_status lg_begin_step(const lg_cache *c, cudaStream_t s) {
  lg_status st = check_cache(c);
  if (st != LG_OK) return st;
  return cuda_status(lg::launch_begin_step(*c, s));
}

lg_status lg_append(const lg_cache *c, int layer0, int n_layers, const void *k_new,
                    const void *v_new, const int32_t *pos_new, const lg_guard_params *p,
                    cudaStream_t s) {
  lg_status st = check_cache(c);
  if (st != LG_OK) return st;
  if ((st = check_params(p)) != LG_OK) return st;
  if (layer0 < 0 || n_layers < 1 || layer0 + n_layers > c->L) return LG_ERR_INVALID_ARG;
  if (!k_new || !v_new || !aligned16(k_new) || !aligned16(v_new)) return LG_ERR_INVALID_ARG;
  if (c->pos && !pos_new) return LG_ERR_INVALID_ARG;
  return cuda_status(lg::launch_append(*c, layer0, n_layers, k_new, v_new, pos_new,
                                       p->guard_layer, s));
}

lg_status lg_sketch_build(const lg_cache *c, const lg_guard_params *p, int max_len,
                          cudaStream_t s) {
  lg_status st = check_cache(c);
  if (st != LG_OK) return st;
  if ((st = check_params(p)) != LG_OK) return st;
  if (!c->sketch || p->guard_layer < 0 || p->guard_layer >= c->L || max_len < 0)
    return LG_ERR_INVALID_ARG;
  return cuda_status(lg::launch_sketch_build(*c, p->guard_layer, max_len, s));
}

lg_status lg_decode_attend(const lg_cache *c, int layer0, int n_layers, const void *q, int H_q,
                           float scale, void *out, float *stats, int suffix_w,
                           int accumulate_h2o, int max_len, void *ws, size_t ws_bytes,
                           cudaStream_t s) {
  lg_status st = check_cache(c);
  if (st != LG_OK) return st;
  if (layer0 < 0 || n_layers < 1 || layer0 + n_layers > c->L) return LG_ERR_INVALID_ARG;
  if (H_q < 1 || H_q % c->H_kv) return LG_ERR_INVALID_ARG;
  const int g = H_q / c->H_kv;
  if (g > 8) return LG_ERR_UNSUPPORTED;
  if (!q || !out || !stats || !aligned16(q) || !aligned16(out) || !aligned16(stats))
    return LG_ERR_INVALID_ARG;
  if (suffix_w < 1 || max_len < 1 || !(scale > 0.f) || !isfinite(scale)) return LG_ERR_INVALID_ARG;
  if (accumulate_h2o && !c->h2o) return LG_ERR_INVALID_ARG;
  const AttendLayout L = attend_layout(c, H_q, n_layers, max_len, accumulate_h2o);
  if (!ws || ((uintptr_t)ws & 255u) || ws_bytes < L.total) return LG_ERR_WORKSPACE;
  lg::AttendArgs a;
  a.K = c->k;
  a.V = c->v;
  a.q = q;
  a.seq_off = c->seq_off;
  a.len = c->len;
  a.status = c->dev_status;
  a.partial = (float *)ws;
  float *final_ml = accumulate_h2o ? (float *)((char *)ws + L.partial_bytes) : nullptr;
  a.logits = accumulate_h2o ? (float *)((char *)ws + L.partial_bytes + L.final_bytes) : nullptr;
  a.counter = (int *)((char *)ws + L.partial_bytes + L.final_bytes + L.logits_bytes);
  a.out = out;
  a.stats = stats;
  a.final_ml = final_ml;
  a.S_total = c->S_total;
  a.layer0 = layer0;
  a.n_layers = n_layers;
  a.batch = c->batch;
  a.H_kv = c->H_kv;
  a.H_q = H_q;
  a.chunk_rows = L.chunk_rows;
  a.max_chunks = L.max_chunks;
  a.max_len = max_len;
  a.suffix_w = suffix_w;
  a.qscale = scale * 1.4426950408889634f;
  const int64_t rows_total = (int64_t)c->L * c->H_kv * c->S_total;
  if (c->dtype == LG_BF16 && rows_total >= ((int64_t)1 << 31)) return LG_ERR_UNSUPPORTED;
  return cuda_status(lg::launch_attend(a, c->dtype, c->d, g, rows_total, out, stats, final_ml,
                                       accumulate_h2o ? c->h2o : nullptr, s));
}

lg_status lg_detect(const lg_cache *c, const float *stats, int H_q, lg_guard_state *state,
                    const int32_t *budget, const lg_guard_params *p, int32_t *flags,
                    int32_t *spans, double *diag, void *dstate, cudaStream_t s) {
  lg_status st = check_cache(c);
  if (st != LG_OK) return st;
  if ((st = check_params(p)) != LG_OK) return st;
  if (!c->sketch || !stats || !state || !budget || !flags || !spans || !dstate)
    return LG_ERR_INVALID_ARG;
  if (((uintptr_t)dstate & 3u) || ((uintptr_t)stats & 15u) || ((uintptr_t)state & 15u))
    return LG_ERR_INVALID_ARG;
  if (H_q < 1 || H_q % c->H_kv) return LG_ERR_INVALID_ARG;
  if (lg::detect_smem_bytes(*p, c->H_kv * c->d / 32) > 200 * 1024) return LG_ERR_UNSUPPORTED;
  return cuda_status(lg::launch_detect(*c, stats, H_q, state, budget, *p, flags, spans, diag,
                                       dstate, nullptr, nullptr, 0, 0, s));
}

lg_status lg_detect_prune(const lg_cache *c, const float *stats, int H_q, lg_guard_state *state,
                          const int32_t *budget, const lg_guard_params *p, int32_t *flags,
                          int32_t *spans, double *diag, void *dstate, int32_t *kept_idx,
                          int32_t *kept_count, int max_keep, int max_len, cudaStream_t s) {
  lg_status st = check_cache(c);
  if (st != LG_OK) return st;
  if ((st = check_params(p)) != LG_OK) return st;
  if (!c->sketch || !stats || !state || !budget || !flags || !spans || !dstate)
    return LG_ERR_INVALID_ARG;
  if (!kept_idx || !kept_count || max_keep < 1 || max_len < 0) return LG_ERR_INVALID_ARG;
  if (((uintptr_t)dstate & 3u) || ((uintptr_t)stats & 15u) || ((uintptr_t)state & 15u))
    return LG_ERR_INVALID_ARG;
  if (H_q < 1 || H_q % c->H_kv) return LG_ERR_INVALID_ARG;
  if (lg::detect_smem_bytes(*p, c->H_kv * c->d / 32) > 200 * 1024) return LG_ERR_UNSUPPORTED;
  st = cuda_status(lg::launch_detect(*c, stats, H_q, state, budget, *p, flags, spans, diag,
                                     dstate, kept_idx, kept_count, max_keep, max_len, s));
  if (st != LG_OK) return st;
  return cuda_status(lg::launch_compact(*c, kept_idx, kept_count, max_keep, s));
}

lg_status lg_default_token_params(lg_token_params *tp) {
  if (!tp) return LG_ERR_INVALID_ARG;
  memset(tp, 0, sizeof(*tp));
  tp->cr_every = 16;
  tp->theta_streak = 6;    // App. B.2
  tp->hist = 512;
  tp->theta_cr = 0.12;     // App. B.2
  tp->theta_conf = 0.9;    // App. B.2
  return LG_OK;
}

size_t lg_token_state_size(const lg_cache *c, const lg_guard_params *p,
                           const lg_token_params *tp) {
  if (check_cache(c) != LG_OK || check_params(p) != LG_OK || check_token_params(p, tp) != LG_OK)
    return 0;
  return (size_t)c->batch * lg::token_state_words(*p, *tp) * sizeof(int32_t);
}

lg_status lg_token_detect(const lg_cache *c, const int32_t *tokens, const float *pmax,
                          const int32_t *kept_idx, const int32_t *kept_count, int max_keep,
                          lg_guard_state *state, const lg_guard_params *p,
                          const lg_token_params *tp, int32_t *flags, int32_t *spans, double *diag,
                          void *tstate, cudaStream_t s) {
  lg_status st = check_cache(c);
  if (st != LG_OK) return st;
  if ((st = check_params(p)) != LG_OK) return st;
  if ((st = check_token_params(p, tp)) != LG_OK) return st;
  if (!tokens || !pmax || !state || !flags || !spans || !tstate) return LG_ERR_INVALID_ARG;
  if (((uintptr_t)state & 15u) || ((uintptr_t)tstate & 7u)) return LG_ERR_INVALID_ARG;
  if ((kept_idx == nullptr) != (kept_count == nullptr) || (kept_idx && max_keep < 1))
    return LG_ERR_INVALID_ARG;
  return cuda_status(lg::launch_token_detect(*c, tokens, pmax, const_cast<int32_t *>(kept_idx),
                                             const_cast<int32_t *>(kept_count), max_keep, state,
                                             *p, *tp, flags, spans, diag, tstate, nullptr, 0, s));
}

lg_status lg_token_detect_prune(const lg_cache *c, const int32_t *tokens, const float *pmax,
                                lg_guard_state *state, const int32_t *budget,
                                const lg_guard_params *p, const lg_token_params *tp,
                                int32_t *flags, int32_t *spans, double *diag, void *tstate,
                                int32_t *kept_idx, int32_t *kept_count, int max_keep,
                                int max_len, cudaStream_t s) {
  lg_status st = check_cache(c);
  if (st != LG_OK) return st;
  if ((st = check_params(p)) != LG_OK) return st;
  if ((st = check_token_params(p, tp)) != LG_OK) return st;
  if (!tokens || !pmax || !state || !budget || !flags || !spans || !tstate)
    return LG_ERR_INVALID_ARG;
  if (((uintptr_t)state & 15u) || ((uintptr_t)tstate & 7u)) return LG_ERR_INVALID_ARG;
  if (!kept_idx || !kept_count || max_keep < 1 || max_len < 0) return LG_ERR_INVALID_ARG;
  st = cuda_status(lg::launch_token_detect(*c, tokens, pmax, kept_idx, kept_count, max_keep,
                                           state, *p, *tp, flags, spans, diag, tstate, budget,
                                           max_len, s));
  if (st != LG_OK) return st;
  return cuda_status(lg::launch_compact(*c, kept_idx, kept_count, max_keep, s));
}

size_t lg_detect_state_size(const lg_cache *c, const lg_guard_params *p) {
  if (check_cache(c) != LG_OK || check_params(p) != LG_OK) return 0;
  return lg::detect_state_bytes(*c, *p);
}

lg_status lg_prune_compact(const lg_cache *c, const int32_t *flags, const int32_t *spans,
                           const lg_guard_state *state, const int32_t *budget,
                           const lg_guard_params *p, int32_t *kept_idx, int32_t *kept_count,
                           int max_keep, int max_len, cudaStream_t s) {
  lg_status st = check_cache(c);
  if (st != LG_OK) return st;
  if ((st = check_params(p)) != LG_OK) return st;
  if (!budget || !kept_idx || !kept_count || max_keep < 1 || max_len < 0) return LG_ERR_INVALID_ARG;
  if (flags && (!spans || !state)) return LG_ERR_INVALID_ARG;
  return cuda_status(lg::launch_prune_compact(*c, flags, spans, state, budget, *p, kept_idx,
                                              kept_count, max_keep, max_len, s));
}

lg_status lg_h2o_reset(const lg_cache *c, int max_len, cudaStream_t s) {
  lg_status st = check_cache(c);
  if (st != LG_OK) return st;
  if (!c->h2o || max_len < 0) return LG_ERR_INVALID_ARG;
  return cuda_status(lg::launch_h2o_reset(*c, max_len, s));
}

lg_status lg_h2o_evict(const lg_cache *c, const int32_t *budget, const int32_t *pos_now,
                       int max_len, cudaStream_t s) {
  lg_status st = check_cache(c);
  if (st != LG_OK) return st;
  if (!c->h2o || !budget || !pos_now || max_len < 0) return LG_ERR_INVALID_ARG;
  return cuda_status(lg::launch_h2o_evict(*c, budget, pos_now, max_len, s));
}

lg_status lg_streaming_evict(const lg_cache *c, const int32_t *budget, const int32_t *pos_now,
                             int n_sink, int max_len, cudaStream_t s) {
  lg_status st = check_cache(c);
  if (st != LG_OK) return st;
  if (!c->pos || !budget || !pos_now || max_len < 0 || n_sink < 0) return LG_ERR_INVALID_ARG;
  return cuda_status(lg::launch_streaming_evict(*c, budget, pos_now, n_sink, max_len, s));
}

lg_status lg_read_device_status(const lg_cache *c, int32_t *host_code, cudaStream_t s) {
  if (!c || !c->dev_status || !host_code) return LG_ERR_INVALID_ARG;
  if (cudaMemcpyAsync(host_code, c->dev_status, sizeof(int32_t), cudaMemcpyDeviceToHost, s) !=
      cudaSuccess)
    return LG_ERR_CUDA;
  return cuda_status(cudaStreamSynchronize(s));
}

}  // extern "C"
