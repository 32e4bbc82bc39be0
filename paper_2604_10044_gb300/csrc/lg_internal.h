// Internal launch interfaces between the C ABI (lg_api.cu) and the kernel files.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include "lg.h"

namespace lg {

struct AttendArgs {
  const void *K, *V;       // cache [L][H_kv][S_total][d]
  const void *q;           // [n_layers][batch][H_q][d]
  const int64_t *seq_off;  // [batch]
  const int32_t *len;      // [batch]
  int32_t *status;
  float *partial;          // [n_layers][batch][H_q][max_chunks][d + 8]
  float *logits;           // nullable [n_layers][H_kv][S_total][g], log2 units
  int *counter;            // [1 + n_layers * batch * H_kv], zeroed by each call (bf16 pass):
                           // the chunk counter, then chunks done per (layer, sequence, kv-head)
  void *out;               // [n_layers][batch][H_q][d] dtype
  float *stats;            // [n_layers][batch][H_q][4]
  float *final_ml;         // nullable [n_layers][batch][H_q][2]: merged (M, l), log2 units
  int64_t S_total;
  int layer0, n_layers, batch, H_kv, H_q;
  int chunk_rows;          // rows per CTA, a multiple of the tile
  int max_chunks;
  int max_len;
  int suffix_w;
  float qscale;            // softmax scale * log2(e)
};

int attend_tile_rows(int dtype, int d);
cudaError_t launch_attend(const AttendArgs &a, int dtype, int d, int g, int64_t rows_total,
                          void *out, float *stats, float *final_ml, float *h2o, cudaStream_t s);
// tensor-core partial pass for bf16 caches (lg_attend_mma.cu)
int mma_tile_rows();
cudaError_t launch_attend_mma_partial(const AttendArgs &a, int d, int g, int64_t rows_total,
                                      cudaStream_t s);

// guard kernels (lg_guard.cu)
cudaError_t launch_begin_step(const lg_cache &c, cudaStream_t s);
cudaError_t launch_append(const lg_cache &c, int layer0, int n_layers, const void *k_new,
                          const void *v_new, const int32_t *pos_new, int guard_layer,
                          cudaStream_t s);
cudaError_t launch_sketch_build(const lg_cache &c, int guard_layer, int max_len, cudaStream_t s);
cudaError_t launch_state_init(const lg_cache &c, lg_guard_state *state, int t_gen0,
                              cudaStream_t s);
// kept_idx nullable: when set, the retained set is formed in the same kernel (no compaction)
cudaError_t launch_detect(const lg_cache &c, const float *stats, int H_q, lg_guard_state *state,
                          const int32_t *budget, const lg_guard_params &p, int32_t *flags,
                          int32_t *spans, double *diag, void *dstate, int32_t *kept_idx,
                          int32_t *kept_count, int max_keep, int max_len, cudaStream_t s);
size_t detect_state_bytes(const lg_cache &c, const lg_guard_params &p);
int detect_smem_rows(const lg_guard_params &p);
size_t detect_smem_bytes(const lg_guard_params &p, int nwords);
cudaError_t launch_prune_compact(const lg_cache &c, const int32_t *flags, const int32_t *spans,
                                 const lg_guard_state *state, const int32_t *budget,
                                 const lg_guard_params &p, int32_t *kept_idx,
                                 int32_t *kept_count, int max_keep, int max_len, cudaStream_t s);
cudaError_t launch_compact(const lg_cache &c, const int32_t *kept_idx, const int32_t *kept_count,
                           int max_keep, cudaStream_t s);
// token-level monitor (lg_token.cu)
size_t token_state_words(const lg_guard_params &p, const lg_token_params &tp);
size_t token_smem_bytes(const lg_guard_params &p, const lg_token_params &tp);
// budget non-null: the kernel also writes this step's kept lists over kept_idx/kept_count
cudaError_t launch_token_detect(const lg_cache &c, const int32_t *tokens, const float *pmax,
                                int32_t *kept_idx, int32_t *kept_count, int max_keep,
                                lg_guard_state *state, const lg_guard_params &p,
                                const lg_token_params &tp, int32_t *flags, int32_t *spans,
                                double *diag, void *tstate, const int32_t *budget, int max_len,
                                cudaStream_t s);
cudaError_t launch_h2o_reset(const lg_cache &c, int max_len, cudaStream_t s);
cudaError_t launch_h2o_evict(const lg_cache &c, const int32_t *budget, const int32_t *pos_now,
                             int max_len, cudaStream_t s);
cudaError_t launch_streaming_evict(const lg_cache &c, const int32_t *budget,
                                   const int32_t *pos_now, int n_sink, int max_len,
                                   cudaStream_t s);

}  // namespace lg
