/*
 * lgref.h -- CPU oracle for the LoopGuard decode path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the CPU
 * baseline leg of the benchmark may load this library.  It shares no code with
 * the CUDA path: plain loops, fp64 accumulation, each function restating the
 * paper's definition it follows.
 *
 * Layout conventions (host memory, caller-owned):
 *   rows of one (layer, kv-head, sequence) stream: [n][d] in the cache dtype
 *   dtype 0 = bf16 (raw uint16 bits), 1 = fp32
 *   stats per (layer, query head): {m, l, H, S}
 *     m = max_i s_i, l = sum_i exp(s_i - m), H = -sum_i a_i ln a_i,
 *     S = sum over the last W_s rows of a_i, W_s = min(suffix_w, n)
 *
 * Parity pins for every function live in tests/test_oracle_*.py.
 */
#ifndef LGREF_H
#define LGREF_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
  int32_t W;             /* monitor window (Sec. 5.2, App. B.2: 256)          */
  int32_t K;             /* vote threshold of the K-of-3 warning (Eq. 8: 2)   */
  int32_t t_min;         /* warmup (Eq. 9, App. B.2: 64)                      */
  int32_t cooldown;      /* cooldown after an intervention (App. B.2: 32)     */
  int32_t n_anchor;      /* anchor prefix (Sec. 5.3, Sec. 6.1: 32)            */
  int32_t stall_len;     /* theta_stall consecutive steps (App. B.2: 4)       */
  int32_t p_min, p_max;  /* tail-period search range                          */
  int32_t l_min;         /* minimum verified tail length                      */
  int32_t m_rep;         /* verified tail covers m_rep periods                */
  int32_t suffix_w;      /* W_s, suffix width of the attention-mass statistic */
  int32_t guard_layer;   /* layer whose V rows feed the row sketches          */
  int32_t level_max;     /* cap of the aggressiveness level                   */
  int32_t retrig_window; /* a re-trigger within this many steps raises the level */
  int32_t headroom;      /* rows left free below the budget after a prune     */
  int32_t pad;
  double theta_ttr;      /* diversity threshold (App. B.2: 0.2)               */
  double theta_nov;      /* novelty threshold of the stall gate (App. B.2: 0.02) */
  double theta_ent;      /* normalised-entropy threshold                      */
  double theta_lift;     /* suffix-lift threshold                             */
  double tau_ham;        /* row match: Hamming distance <= floor(tau_ham * bits) */
} lgref_params;

typedef struct {
  int32_t t_gen;         /* decode steps seen                                 */
  int32_t cd;            /* cooldown counter cd(t)                            */
  int32_t level;         /* aggressiveness level                              */
  int32_t last_trig;     /* t_gen of the last intervention                    */
  int32_t n_int;         /* interventions so far                              */
  int32_t pad[3];
} lgref_state;

/* Sec. 3.1, Eq. 1 over one kv-head's rows for its g query heads.
   q [g][d], K/V [n][d] (cache dtype); out [g][d], stats [g][4]; alpha [g][n] nullable.
   Returns 0, or -1 when n < 1 or d < 1. */
int lgref_attend_group(int dtype, int d, int n, const void *K, const void *V, int g,
                       const void *q, double scale, int suffix_w, double *out, double *stats,
                       double *alpha);

/* Eq. 1 for every (layer, sequence, kv-head) of a cache laid out [L][H_kv][S_total][d].
   q [L][batch][H_q][d]; out [L][batch][H_q][d]; stats [L][batch][H_q][4];
   h2o nullable [L][H_kv][S_total]: accumulated attention (sum over the GQA group).
   Returns the number of threads used, or -1 on invalid arguments. */
int lgref_attend_all(int dtype, int L, int H_kv, int H_q, int d, int batch, int64_t S_total,
                     const int64_t *seq_off, const int32_t *len, const void *K, const void *V,
                     const void *q, double scale, int suffix_w, double *out, double *stats,
                     double *h2o);

/* sign bits of one row of nelem values: bit j of word w is the sign bit of element 32w + j */
void lgref_sketch(int dtype, int nelem, const void *row, uint32_t *words);

/* 1 iff popcount(a xor b) <= thr over nwords words */
int lgref_match(const uint32_t *a, const uint32_t *b, int nwords, int thr);

/* The loop-onset test (Sec. 5.2, Eq. 8, Eq. 9) for one sequence of length n.
   stats [L][H_q][4]; sketch [n][nwords] (row i = slot i); budget B of the sequence.
   Updates *st; writes flag and span[2] = [lo, hi) of I_bad (empty: [0, 0)).
   diag (nullable, 10 doubles): ebar, lbar, ttr, sig1, sig2, sig3, warn, stall, P*, trigger.
   Returns 0, or -1 on invalid arguments. */
int lgref_detect(int L, int H_q, const double *stats, int n, const uint32_t *sketch, int nwords,
                 int budget, const lgref_params *p, lgref_state *st, int32_t *flag,
                 int32_t *span, double *diag);

/* I_keep (Sec. 5.3, Eq. 10, Eq. 11) for one sequence: kept[] ascending slot indices, returns |I_keep|
   (n when the sequence is not pruned), or -1 when the budget is too small. */
int lgref_keep_set(int n, int budget, int flag, int span_lo, int span_hi, int level,
                   const lgref_params *p, int32_t *kept);

/* index-gather of kept rows (Sec. 5.3): rows[j] <- rows[kept[j]], j < count */
void lgref_compact_rows(void *rows, size_t row_bytes, const int32_t *kept, int count);

/* H2O comparator: rows kept when a (layer, kv-head) stream of n > budget rows is cut to
   `budget`: the budget/2 most recent positions plus the highest accumulated scores.
   kept[] ascending slots; returns the count (n when n <= budget). */
int lgref_h2o_select(int n, const double *score, const int32_t *pos, int budget, int32_t pos_now,
                     int32_t *kept);

/* H2O comparator, one row over budget: the evicted slot (lowest score outside the recent
   window, older position first on ties), or -1 when nothing is evictable. */
int lgref_h2o_argmin(int n, const double *score, const int32_t *pos, int budget, int32_t pos_now);

/* StreamingLLM comparator (attention sinks + sliding window, Sec. 2.2, Sec. 6.1): rows kept when a
   (layer, kv-head) stream of n > budget rows is cut to `budget`: positions < n_sink and the
   budget - n_sink most recent positions.  kept[] ascending slots; returns the count. */
int lgref_streaming_select(int n, const int32_t *pos, int budget, int n_sink, int32_t pos_now,
                           int32_t *kept);

/* StreamingLLM comparator, one row over budget: the slot of the oldest position >= n_sink. */
int lgref_streaming_oldest(int n, const int32_t *pos, int n_sink);

/* ---- token-level monitor (Sec. 5.2, Eq. 8, Eq. 9, App. B.2) on generated token ids ---- */

typedef struct {
  int32_t cr_every;      /* the compression ratio is evaluated every cr_every tokens      */
  int32_t theta_streak;  /* confidence-collapse streak, steps (App. B.2: 6)                */
  int32_t hist;          /* generated tokens the span extension may reach back over        */
  int32_t pad;
  double theta_cr;       /* redundancy threshold (App. B.2: 0.12)                           */
  double theta_conf;     /* top-1 probability threshold (App. B.2: 0.9)                     */
} lgref_token_params;

typedef struct {
  int32_t streak;        /* consecutive steps with p_max > theta_conf                       */
  int32_t synced;        /* cache length seen by the previous step (-1 before the first)    */
  int32_t appended;      /* trailing cache rows that are consecutive generated tokens       */
  int32_t pad;
  double cr;             /* the last evaluated compression ratio                            */
} lgref_token_state;

/* Phrases of the greedy LZ77 parse of x[0..w): at each position the longest earlier match
   (overlap allowed, up to the end) becomes one phrase when it covers at least 2 tokens, else
   the token is one literal phrase. */
int lgref_lz77_phrases(const int32_t *x, int w);

/* One decode step of the token-level monitor.  tokens[0..T) are every generated token so far
   (tokens[T-1] is this step's), pmax this step's top-1 probability, n the cache length after
   this step's append; kept[0..kept_count) (nullable; kept_count -1 = no prune) the retained
   slots of the prune that followed the previous step.  Writes the trigger flag and the span
   [lo, hi) of cache slots (empty [0,0) without a tail period) and updates the guard and
   monitor state.  diag nullable [10]: {ttr, cr, streak, vote1, vote2, vote3, warn, stall, P*,
   trigger}. */
int lgref_token_detect(const int32_t *tokens, int T, double pmax, int n, const int32_t *kept,
                       int kept_count, const lgref_params *p, const lgref_token_params *tp,
                       lgref_state *st, lgref_token_state *ts, int32_t *flag, int32_t *span,
                       double *diag);

#ifdef __cplusplus
}
#endif
#endif
