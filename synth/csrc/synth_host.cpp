// Host side of the synthetic workload generator (harness).  Same recipe and
// same source of truth as the device side: synth_core.h.  Build with
// -ffp-contract=off so that no multiply-add is fused.
#include <string.h>

#include "synth_core.h"

extern "C" {

static void store(const syn_workload *w, void *out, int64_t i, float v) {
  if (w->dtype == SYN_BF16)
    ((uint16_t *)out)[i] = syn_bf16_bits(v);
  else
    ((float *)out)[i] = v;
}

/* rows [p0, p0 + count) of one (layer, kv-head, sequence) stream, [count][d] in the cache dtype */
void syn_host_rows(const syn_workload *w, const syn_seq *s, int is_value, int layer, int kvh,
                   int seq, int64_t p0, int64_t count, void *out) {
  for (int64_t r = 0; r < count; ++r)
    for (int e = 0; e < w->d; ++e)
      store(w, out, r * w->d + e, syn_row_value(w, s, is_value, layer, kvh, seq, p0 + r, e));
}

/* K and V [L][H_kv][S_total][d]: rows [0, n_rows[b]) at slots seq_off[b] + p */
void syn_host_fill_cache(const syn_workload *w, const syn_seq *seqs, int batch,
                         const int64_t *seq_off, const int32_t *n_rows, int64_t S_total, void *K,
                         void *V) {
  const int64_t esz = w->dtype == SYN_BF16 ? 2 : 4;
#pragma omp parallel for collapse(2) schedule(dynamic)
  for (int lh = 0; lh < w->L * w->H_kv; ++lh)
    for (int b = 0; b < batch; ++b) {
      int layer = lh / w->H_kv, kvh = lh % w->H_kv;
      int64_t base = ((int64_t)lh * S_total + seq_off[b]) * w->d * esz;
      syn_host_rows(w, &seqs[b], 0, layer, kvh, b, 0, n_rows[b], (char *)K + base);
      syn_host_rows(w, &seqs[b], 1, layer, kvh, b, 0, n_rows[b], (char *)V + base);
    }
}

/* One decode step's inputs for the tokens at positions pos[b]:
   q [L][batch][H_q][d], k_new / v_new [L][batch][H_kv][d], all in the cache dtype. */
void syn_host_step(const syn_workload *w, const syn_seq *seqs, int batch, const int64_t *pos,
                   void *q, void *k_new, void *v_new) {
#pragma omp parallel for collapse(2)
  for (int layer = 0; layer < w->L; ++layer)
    for (int b = 0; b < batch; ++b) {
      float qv[512];
      for (int h = 0; h < w->H_q; ++h) {
        syn_query(w, &seqs[b], layer, h, b, pos[b], qv);
        int64_t o = (((int64_t)layer * batch + b) * w->H_q + h) * w->d;
        for (int e = 0; e < w->d; ++e) store(w, q, o + e, qv[e]);
      }
      for (int kvh = 0; kvh < w->H_kv; ++kvh) {
        int64_t o = (((int64_t)layer * batch + b) * w->H_kv + kvh) * w->d;
        for (int e = 0; e < w->d; ++e) {
          store(w, k_new, o + e, syn_row_value(w, &seqs[b], 0, layer, kvh, b, pos[b], e));
          store(w, v_new, o + e, syn_row_value(w, &seqs[b], 1, layer, kvh, b, pos[b], e));
        }
      }
    }
}

/* a few raw draws, for the generator's own self-test */
void syn_host_normals(uint64_t seed, int role, int layer, int head, int seq, uint64_t idx0,
                      int64_t count, float *out) {
  uint64_t k = syn_key(seed, role, layer, head, seq);
  for (int64_t i = 0; i < count; ++i) out[i] = syn_normal(k, idx0 + (uint64_t)i);
}

uint64_t syn_host_mix(uint64_t x) { return syn_mix(x); }

}  // extern "C"
