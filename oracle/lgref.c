/*
 * lgref.c -- CPU oracle for the LoopGuard decode path.
 *
 * TEST INFRASTRUCTURE ONLY: loaded by the tests, the smoke check and the CPU
 * baseline leg of the benchmark, never by the product path.  Plain loops in
 * fp64; no blocking, fusion or reordering beyond what each definition states.
 * Shares no code, header or table with the CUDA library.
 *
 * Paper: LoopGuard: Breaking Self-Reinforcing Attention Loops via Dynamic KV
 * Cache Intervention (arXiv 2604.10044).
 *   attention over the retained cache ........ Sec. 3.1, Eq. 1
 *   K-of-3 warning vote ...................... Sec. 5.2, Eq. 8
 *   debounced trigger (warmup, cooldown) ..... Sec. 5.2, Eq. 9
 *   stall and suffix self-alignment gates .... Sec. 5.2, App. B.2
 *   retained set I_keep, tail-cleaned recent . Sec. 5.3, Eq. 10, Eq. 11
 *   progressive aggressiveness, gather ....... Sec. 5.3
 *   H2O comparator (cited, not defined) ...... Sec. 2.2, Sec. 6.1
 *   StreamingLLM comparator (cited) .......... Sec. 2.2, Sec. 6.1
 *   token-level monitor (TTR, CR, p_max) ..... Sec. 4.3, Sec. 5.2, Eq. 8, Eq. 9, App. B.2
 *
 * The paper's detector reads generated token ids and top-1 probabilities:
 * lgref_token_detect follows it on those inputs.  A decode path that carries
 * only K/V caches and attention has neither, so lgref_detect restates each
 * signal over attention statistics and sign sketches of the guard layer's V
 * rows.  Where the paper is silent the constants are chosen here, stated
 * beside each function; tests/test_oracle_*.py pin every function.
 */
#include "lgref.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ---------------------------------------------------------------- values */

static double widen(int dtype, const void *base, int64_t i) {
  if (dtype == 0) {
    uint32_t bits = (uint32_t)((const uint16_t *)base)[i] << 16;
    float f;
    memcpy(&f, &bits, 4);
    return (double)f;
  }
  return (double)((const float *)base)[i];
}

/* ---------------------------------------------------------------- Eq. 1 */

int lgref_attend_group(int dtype, int d, int n, const void *K, const void *V, int g,
                       const void *q, double scale, int suffix_w, double *out, double *stats,
                       double *alpha) {
  if (n < 1 || d < 1 || g < 1) return -1;
  double *s = (double *)malloc(sizeof(double) * (size_t)n);
  double *a = (double *)malloc(sizeof(double) * (size_t)n);
  if (!s || !a) {
    free(s);
    free(a);
    return -1;
  }
  int Ws = suffix_w < n ? suffix_w : n;
  for (int h = 0; h < g; ++h) {
    /* logits s_i = <q, k_i> / sqrt(d_h) (the caller passes scale) */
    for (int i = 0; i < n; ++i) {
      double dot = 0.0;
      for (int e = 0; e < d; ++e)
        dot += widen(dtype, q, (int64_t)h * d + e) * widen(dtype, K, (int64_t)i * d + e);
      s[i] = dot * scale;
    }
    /* softmax over the retained rows */
    double m = s[0];
    for (int i = 1; i < n; ++i)
      if (s[i] > m) m = s[i];
    double l = 0.0;
    for (int i = 0; i < n; ++i) l += exp(s[i] - m);
    for (int i = 0; i < n; ++i) a[i] = exp(s[i] - m) / l;
    /* head output o = sum_i a_i v_i */
    for (int e = 0; e < d; ++e) {
      double o = 0.0;
      for (int i = 0; i < n; ++i) o += a[i] * widen(dtype, V, (int64_t)i * d + e);
      out[(int64_t)h * d + e] = o;
    }
    /* statistics: entropy of the attention row, mass on the last W_s rows */
    double H = 0.0;
    for (int i = 0; i < n; ++i)
      if (a[i] > 0.0) H -= a[i] * log(a[i]);
    double S = 0.0;
    for (int i = n - Ws; i < n; ++i) S += a[i];
    stats[4 * h + 0] = m;
    stats[4 * h + 1] = l;
    stats[4 * h + 2] = H;
    stats[4 * h + 3] = S;
    if (alpha)
      for (int i = 0; i < n; ++i) alpha[(int64_t)h * n + i] = a[i];
  }
  free(s);
  free(a);
  return 0;
}

int lgref_attend_all(int dtype, int L, int H_kv, int H_q, int d, int batch, int64_t S_total,
                     const int64_t *seq_off, const int32_t *len, const void *K, const void *V,
                     const void *q, double scale, int suffix_w, double *out, double *stats,
                     double *h2o) {
  if (L < 1 || H_kv < 1 || H_q % H_kv || d < 1 || batch < 1) return -1;
  const int g = H_q / H_kv;
  const int64_t esz = dtype == 0 ? 2 : 4;
  const int ngroups = L * batch * H_kv;
  int threads = 1;
  int bad = 0;
#pragma omp parallel
  {
#ifdef _OPENMP
#pragma omp single
    threads = omp_get_num_threads();
#endif
#pragma omp for schedule(dynamic)
    for (int t = 0; t < ngroups; ++t) {
      int kvh = t % H_kv, b = (t / H_kv) % batch, layer = t / (H_kv * batch);
      int n = len[b];
      int64_t row0 = ((int64_t)layer * H_kv + kvh) * S_total + seq_off[b];
      const char *Kb = (const char *)K + row0 * d * esz;
      const char *Vb = (const char *)V + row0 * d * esz;
      int64_t qh0 = ((int64_t)layer * batch + b) * H_q + (int64_t)kvh * g;
      const char *qb = (const char *)q + qh0 * d * esz;
      double *alpha = h2o ? (double *)malloc(sizeof(double) * (size_t)g * (size_t)n) : NULL;
      int rc = lgref_attend_group(dtype, d, n, Kb, Vb, g, qb, scale, suffix_w, out + qh0 * d,
                                  stats + qh0 * 4, alpha);
      if (rc) bad = 1;
      if (h2o && alpha && !rc) {
        /* H2O accumulated score: attention received, summed over the heads sharing the row */
        double *sc = h2o + row0;
        for (int i = 0; i < n; ++i)
          for (int h = 0; h < g; ++h) sc[i] += alpha[(int64_t)h * n + i];
      }
      free(alpha);
    }
  }
  return bad ? -1 : threads;
}

/* ---------------------------------------------------------------- sketches */

void lgref_sketch(int dtype, int nelem, const void *row, uint32_t *words) {
  for (int w = 0; w < nelem / 32; ++w) words[w] = 0;
  for (int j = 0; j < nelem; ++j) {
    uint32_t sign;
    if (dtype == 0)
      sign = ((const uint16_t *)row)[j] >> 15;
    else {
      uint32_t bits;
      memcpy(&bits, (const float *)row + j, 4);
      sign = bits >> 31;
    }
    words[j / 32] |= sign << (j % 32);
  }
}

int lgref_match(const uint32_t *a, const uint32_t *b, int nwords, int thr) {
  int dist = 0;
  for (int w = 0; w < nwords; ++w) {
    uint32_t x = a[w] ^ b[w];
    for (int bit = 0; bit < 32; ++bit) dist += (x >> bit) & 1u;
  }
  return dist <= thr;
}

/* ---------------------------------------------------------------- Sec. 5.2 */

int lgref_detect(int L, int H_q, const double *stats, int n, const uint32_t *sketch, int nwords,
                 int budget, const lgref_params *p, lgref_state *st, int32_t *flag,
                 int32_t *span, double *diag) {
  if (L < 1 || H_q < 1 || n < 0 || nwords < 1 || !p || !st) return -1;
  const int thr = (int)floor(p->tau_ham * (double)(nwords * 32));
#define ROW(i) (sketch + (int64_t)(i) * nwords)
  int sig1 = 0, sig2 = 0, sig3 = 0, stall = 0, tailrep = 0, Pstar = 0;
  double ebar = 1.0, lbar = 0.0, ttr = 1.0;
  if (n >= 1) {
    /* concentration: mean normalised entropy over every layer and head */
    double acc = 0.0;
    for (int t = 0; t < L * H_q; ++t) acc += n >= 2 ? stats[4 * t + 2] / log((double)n) : 1.0;
    ebar = acc / (double)(L * H_q);
    /* locking: mean suffix lift S * n / W_s (1 for uniform attention) */
    int Ws = p->suffix_w < n ? p->suffix_w : n;
    acc = 0.0;
    for (int t = 0; t < L * H_q; ++t) acc += stats[4 * t + 3] * (double)n / (double)Ws;
    lbar = acc / (double)(L * H_q);

    /* diversity: fraction of novel rows in the window W_t of the last min(W, n) rows */
    int w = p->W < n ? p->W : n;
    int lo = n - w;
    int n_novel = 0, novel_tail = 0;
    for (int i = lo; i < n; ++i) {
      int novel = 1;
      for (int j = lo; j < i; ++j)
        if (lgref_match(ROW(i), ROW(j), nwords, thr)) {
          novel = 0;
          break;
        }
      n_novel += novel;
      if (i >= n - p->stall_len) novel_tail += novel;
    }
    ttr = (double)n_novel / (double)w;
    /* novelty stagnation: novel fraction over the last theta_stall rows below theta_nov */
    if (w >= p->stall_len && p->stall_len > 0)
      stall = (double)novel_tail / (double)p->stall_len < p->theta_nov;

    /* suffix self-alignment: smallest period P whose last max(m_rep P, l_min) rows each
       match the row P earlier */
    for (int P = p->p_min; P <= p->p_max && !tailrep; ++P) {
      int span_len = p->m_rep * P > p->l_min ? p->m_rep * P : p->l_min;
      if (n < span_len + P) continue;
      int all = 1;
      for (int i = n - span_len; i < n && all; ++i) all = lgref_match(ROW(i), ROW(i - P), nwords, thr);
      if (all) {
        tailrep = 1;
        Pstar = P;
      }
    }
    sig1 = ttr < p->theta_ttr;
    sig2 = ebar < p->theta_ent;
    sig3 = lbar >= p->theta_lift;
  }
  int warn = sig1 + sig2 + sig3 >= p->K;
  int trigger = st->t_gen >= p->t_min && st->cd == 0 && warn && (stall || tailrep);

  span[0] = 0;
  span[1] = 0;
  if (trigger && tailrep) {
    /* I_bad: every copy of the verified tail period, extended back while rows keep matching
       the row P* earlier, clipped to the recent window W^recent = [n - R, n) */
    int R = budget / 2;
    int span_len = p->m_rep * Pstar > p->l_min ? p->m_rep * Pstar : p->l_min;
    int lo_ext = Pstar > n - R ? Pstar : n - R;
    int s = n - span_len;
    if (s < lo_ext)
      s = lo_ext;
    else
      while (s - 1 >= lo_ext && lgref_match(ROW(s - 1), ROW(s - 1 - Pstar), nwords, thr)) --s;
    int bad_lo = s - Pstar > n - R ? s - Pstar : n - R;
    if (bad_lo < 0) bad_lo = 0;
    span[0] = bad_lo;
    span[1] = n;
  }
  *flag = trigger;

  /* guard state: progressive level on a quick re-trigger, cooldown, step counter */
  if (trigger) {
    int quick = st->t_gen - st->last_trig <= p->retrig_window;
    st->level = quick ? (st->level + 1 < p->level_max ? st->level + 1 : p->level_max) : 0;
    st->last_trig = st->t_gen;
    st->cd = p->cooldown;
    st->n_int += 1;
  } else if (st->cd > 0) {
    st->cd -= 1;
  }
  st->t_gen += 1;

  if (diag) {
    diag[0] = ebar;
    diag[1] = lbar;
    diag[2] = ttr;
    diag[3] = sig1;
    diag[4] = sig2;
    diag[5] = sig3;
    diag[6] = warn;
    diag[7] = stall;
    diag[8] = tailrep ? Pstar : 0;
    diag[9] = trigger;
  }
#undef ROW
  return 0;
}

/* ---------------------------------------------------------------- Sec. 5.3 */

int lgref_keep_set(int n, int budget, int flag, int span_lo, int span_hi, int level,
                   const lgref_params *p, int32_t *kept) {
  if (n < 0 || !p) return -1;
  if (!flag && n <= budget) {
    for (int i = 0; i < n; ++i) kept[i] = i;
    return n;
  }
  if (!flag) {
    /* budget event: no tail detected, base aggressiveness */
    level = 0;
    span_lo = span_hi = 0;
  }
  int headroom = p->headroom < budget / 4 ? p->headroom : budget / 4;
  int T_keep = budget - headroom;
  int R = budget / 2;
  int B_recent = (budget / 4) >> level;
  int B_sparse = T_keep - p->n_anchor - budget / 4;
  if (B_sparse < 0) return -1;

  unsigned char *mask = (unsigned char *)calloc((size_t)(n > 0 ? n : 1), 1);
  if (!mask) return -1;
  /* anchors: the prefix {0, ..., N_anchor - 1} */
  for (int i = 0; i < n && i < p->n_anchor; ++i) mask[i] = 1;
  /* recent window W^recent = [n - R, n), never reaching into the anchors */
  int rw_lo = n - R > p->n_anchor ? n - R : p->n_anchor;
  if (rw_lo > n) rw_lo = n;
  /* sparse long-range context: uniform subsample of the history outside W^recent */
  int n_c = rw_lo - p->n_anchor;
  if (n_c > 0) {
    if (n_c <= B_sparse)
      for (int i = p->n_anchor; i < rw_lo; ++i) mask[i] = 1;
    else
      for (int j = 0; j < B_sparse; ++j)
        mask[p->n_anchor + (int)(((int64_t)j * n_c) / B_sparse)] = 1;
  }
  /* tail-cleaned recent context: C_recent = W^recent \ I_bad; I_recent = its last
     B_recent(level) rows */
  int taken = 0;
  for (int i = n - 1; i >= rw_lo && taken < B_recent; --i) {
    if (i >= span_lo && i < span_hi) continue;
    mask[i] = 1;
    ++taken;
  }
  int count = 0;
  for (int i = 0; i < n; ++i)
    if (mask[i]) kept[count++] = i;
  free(mask);
  return count;
}

void lgref_compact_rows(void *rows, size_t row_bytes, const int32_t *kept, int count) {
  char *tmp = (char *)malloc(row_bytes * (size_t)(count > 0 ? count : 1));
  if (!tmp) return;
  for (int j = 0; j < count; ++j)
    memcpy(tmp + (size_t)j * row_bytes, (const char *)rows + (size_t)kept[j] * row_bytes,
           row_bytes);
  memcpy(rows, tmp, row_bytes * (size_t)count);
  free(tmp);
}

/* ---------------------------------------------------------------- H2O comparator */

typedef struct {
  double score;
  int32_t pos;
  int32_t slot;
} cand_t;

/* ascending (score, pos): the front of the order is evicted first */
static int cand_cmp(const void *x, const void *y) {
  const cand_t *a = (const cand_t *)x, *b = (const cand_t *)y;
  if (a->score < b->score) return -1;
  if (a->score > b->score) return 1;
  return (a->pos > b->pos) - (a->pos < b->pos);
}

int lgref_h2o_select(int n, const double *score, const int32_t *pos, int budget, int32_t pos_now,
                     int32_t *kept) {
  if (n <= budget) {
    for (int i = 0; i < n; ++i) kept[i] = i;
    return n;
  }
  int R = budget / 2;
  unsigned char *keep = (unsigned char *)calloc((size_t)n, 1);
  cand_t *c = (cand_t *)malloc(sizeof(cand_t) * (size_t)n);
  if (!keep || !c) {
    free(keep);
    free(c);
    return -1;
  }
  int n_recent = 0, n_c = 0;
  for (int i = 0; i < n; ++i) {
    if (pos[i] > pos_now - R) {
      keep[i] = 1;
      ++n_recent;
    } else {
      c[n_c].score = score[i];
      c[n_c].pos = pos[i];
      c[n_c].slot = i;
      ++n_c;
    }
  }
  int heavy = budget - n_recent;
  if (heavy < 0) heavy = 0;
  if (heavy > n_c) heavy = n_c;
  qsort(c, (size_t)n_c, sizeof(cand_t), cand_cmp);
  for (int k = n_c - heavy; k < n_c; ++k) keep[c[k].slot] = 1;
  int count = 0;
  for (int i = 0; i < n; ++i)
    if (keep[i]) kept[count++] = i;
  free(keep);
  free(c);
  return count;
}

int lgref_h2o_argmin(int n, const double *score, const int32_t *pos, int budget, int32_t pos_now) {
  int R = budget / 2;
  int best = -1;
  for (int i = 0; i < n; ++i) {
    if (pos[i] > pos_now - R) continue;
    if (best < 0 || score[i] < score[best] || (score[i] == score[best] && pos[i] < pos[best]))
      best = i;
  }
  return best;
}

/* ---------------------------------------------------------------- StreamingLLM comparator */

int lgref_streaming_select(int n, const int32_t *pos, int budget, int n_sink, int32_t pos_now,
                           int32_t *kept) {
  if (n <= budget) {
    for (int i = 0; i < n; ++i) kept[i] = i;
    return n;
  }
  int window = budget - n_sink;
  int count = 0;
  for (int i = 0; i < n; ++i)
    if (pos[i] < n_sink || pos[i] > pos_now - window) kept[count++] = i;
  return count;
}

int lgref_streaming_oldest(int n, const int32_t *pos, int n_sink) {
  int best = -1;
  for (int i = 0; i < n; ++i) {
    if (pos[i] < n_sink) continue;
    if (best < 0 || pos[i] < pos[best]) best = i;
  }
  return best;
}

/* ---------------------------------------------------------------- token-level monitor */

int lgref_lz77_phrases(const int32_t *x, int w) {
  int phrases = 0;
  for (int i = 0; i < w;) {
    int best = 0;
    for (int j = 0; j < i; ++j) {
      int k = 0;
      while (i + k < w && x[j + k] == x[i + k]) ++k;
      if (k > best) best = k;
    }
    ++phrases;
    i += best >= 2 ? best : 1;
  }
  return phrases;
}

int lgref_token_detect(const int32_t *tokens, int T, double pmax, int n, const int32_t *kept,
                       int kept_count, const lgref_params *p, const lgref_token_params *tp,
                       lgref_state *st, lgref_token_state *ts, int32_t *flag, int32_t *span,
                       double *diag) {
  if (T < 1 || n < 1 || !p || !tp || !st || !ts || tp->cr_every < 1) return -1;
  const int32_t *y = tokens;
  const int t = T - 1; /* this step's token */

  /* cache rows that are consecutive generated tokens, this step's row included */
  if (ts->synced >= 0 && kept && kept_count >= 0 && n == kept_count + 1) {
    /* the cache was pruned after the previous step: the kept rows that end the kept list
       one after another, up to the old last row, and were consecutive tokens before, still
       are */
    int run = 0;
    for (int j = kept_count - 1; j >= 0; --j) {
      if (kept[j] != ts->synced - (kept_count - j) || kept[j] < ts->synced - ts->appended) break;
      ++run;
    }
    ts->appended = run + 1;
  } else {
    /* one more after an append; only this step's row after any other change */
    ts->appended = (ts->synced >= 0 && n == ts->synced + 1) ? ts->appended + 1 : 1;
  }
  if (ts->appended > n) ts->appended = n;
  ts->synced = n;

  /* the window W_t: the last min(W, T) generated tokens */
  const int w = p->W < T ? p->W : T;
  const int lo = T - w;
  /* diversity (TTR): distinct tokens of the window over its length; a token is novel when no
     earlier token of the window equals it */
  int n_distinct = 0, novel_tail = 0;
  for (int i = lo; i < T; ++i) {
    int novel = 1;
    for (int j = lo; j < i && novel; ++j) novel = y[j] != y[i];
    n_distinct += novel;
    if (i >= T - p->stall_len) novel_tail += novel;
  }
  const double ttr = (double)n_distinct / (double)w;
  /* redundancy (CR): LZ77 phrases of the window over its length, evaluated every cr_every
     tokens and held in between */
  if (t % tp->cr_every == 0) ts->cr = (double)lgref_lz77_phrases(y + lo, w) / (double)w;
  /* confidence collapse: consecutive steps with p_max above theta_conf */
  ts->streak = pmax > tp->theta_conf ? ts->streak + 1 : 0;
  /* novelty stagnation: novel fraction of the last theta_stall tokens below theta_nov */
  int stall = 0;
  if (w >= p->stall_len && p->stall_len > 0)
    stall = (double)novel_tail / (double)p->stall_len < p->theta_nov;
  /* suffix self-alignment: smallest period P whose last max(m_rep P, l_min) tokens each equal
     the token P earlier */
  int tailrep = 0, Pstar = 0;
  for (int P = p->p_min; P <= p->p_max && !tailrep; ++P) {
    int span_len = p->m_rep * P > p->l_min ? p->m_rep * P : p->l_min;
    if (T < span_len + P) continue;
    int all = 1;
    for (int i = T - span_len; i < T && all; ++i) all = y[i] == y[i - P];
    if (all) {
      tailrep = 1;
      Pstar = P;
    }
  }
  const int sig1 = ttr < p->theta_ttr;
  const int sig2 = ts->cr < tp->theta_cr;
  const int sig3 = ts->streak >= tp->theta_streak;
  const int warn = sig1 + sig2 + sig3 >= p->K;
  const int trigger = st->t_gen >= p->t_min && st->cd == 0 && warn && (stall || tailrep);

  span[0] = 0;
  span[1] = 0;
  if (trigger && tailrep) {
    /* the repetitive tail in generated tokens: the verified run extended back while tokens
       keep equalling the token P* earlier (within the kept history), plus its first period;
       mapped onto the trailing cache rows that hold consecutive generated tokens */
    int span_len = p->m_rep * Pstar > p->l_min ? p->m_rep * Pstar : p->l_min;
    int lim = T - tp->hist > 0 ? T - tp->hist : 0;
    int s = T - span_len;
    while (s - 1 - Pstar >= lim && y[s - 1] == y[s - 1 - Pstar]) --s;
    int bad = T - (s - Pstar);
    if (bad > ts->appended) bad = ts->appended;
    span[0] = n - bad;
    span[1] = n;
  }
  *flag = trigger;

  if (trigger) {
    int quick = st->t_gen - st->last_trig <= p->retrig_window;
    st->level = quick ? (st->level + 1 < p->level_max ? st->level + 1 : p->level_max) : 0;
    st->last_trig = st->t_gen;
    st->cd = p->cooldown;
    st->n_int += 1;
  } else if (st->cd > 0) {
    st->cd -= 1;
  }
  st->t_gen += 1;

  if (diag) {
    diag[0] = ttr;
    diag[1] = ts->cr;
    diag[2] = ts->streak;
    diag[3] = sig1;
    diag[4] = sig2;
    diag[5] = sig3;
    diag[6] = warn;
    diag[7] = stall;
    diag[8] = tailrep ? Pstar : 0;
    diag[9] = trigger;
  }
  return 0;
}
