// Token-level loop-onset monitor (LoopGuard Sec. 5.2, Eq. 8, Eq. 9, App. B.2; indicators of
// Sec. 4.3) over the generated token ids and top-1 probabilities the caller passes each step.
//
// One CTA per sequence.  The monitor state (tstate) of a sequence keeps the last `hist` tokens
// and, for each, the latest earlier equal token of the window as it was when the token arrived
// (a token of the current window [wlo, t] is novel iff that match lies below wlo, so TTR and
// the stall gate cost one comparison of the new token against the window per step), the
// trailing run of every period, the p_max streak, the last compression ratio and the number of
// trailing cache rows that are consecutive generated tokens (to map a token span onto slots).
//   vote 1  TTR = novel tokens of the window / window                 < theta_ttr
//   vote 2  CR  = greedy LZ77 phrases of the window / window           < theta_cr
//           (every cr_every tokens; a phrase is the longest earlier match of >= 2 tokens,
//           overlap allowed, else one literal token)
//   vote 3  consecutive steps with p_max > theta_conf                 >= theta_streak
//   Stall   novel fraction of the last theta_stall tokens             < theta_nov
//   TailRep smallest P in [p_min, p_max] whose last max(m_rep P, l_min) tokens each equal the
//           token P earlier
//   Trigger t_gen >= t_min and cd = 0 and votes >= K and (Stall or TailRep)
// On a trigger with TailRep the span is the verified run extended back while tokens keep
// equalling the token P* earlier (within the kept history), plus its first period, mapped onto
// the trailing cache rows that hold consecutive generated tokens (kept across a prune when the
// caller passes the prune's retained lists).
#include <cuda_runtime.h>
#include <stdint.h>

#include "lg_common.cuh"
#include "lg_internal.h"
#include "lg_keep.cuh"

namespace lg {

namespace {

constexpr int kTokThreads = 256;
constexpr int kTokWarps = kTokThreads / 32;
constexpr int kHdrWords = 16;  // count, streak, synced + 1, appended, cr (2 words), reserved

struct TokenArgs {
  lg_cache c;
  const int32_t *tokens;  // [batch] this step's token of each sequence
  const float *pmax;      // [batch] this step's top-1 probability
  int32_t *kept_idx;    // nullable [batch][max_keep]: the prune after the previous step
  int32_t *kept_count;  // nullable [batch], -1 = that sequence was not pruned
  int max_keep;
  // set: the same CTA goes on to this step's retained set (as lg_prune_compact's kernel forms
  // it), written over the previous kept lists once they have been read
  const int32_t *budget;
  int max_len;
  int prune;
  lg_guard_state *state;
  lg_guard_params p;
  lg_token_params tp;
  int32_t *flags, *spans;
  double *diag;
  int32_t *tstate;
};

// words of one sequence's monitor state, a multiple of 4 (the stored ratio is a double)
__host__ __device__ __forceinline__ int64_t state_stride(int hist, int np) {
  return ((int64_t)kHdrWords + 2 * (int64_t)hist + np + 3) / 4 * 4;
}

__global__ void __launch_bounds__(kTokThreads, 1) token_detect_kernel(TokenArgs a) {
  pdl_enter();
  extern __shared__ __align__(16) int32_t sm[];
  __shared__ int w_latest[kTokWarps], w_nov[kTokWarps], w_tail[kTokWarps], w_pstar[kTokWarps],
      w_run[kTokWarps];
  __shared__ int s_mismatch, s_trig, s_P, s_n_tok, s_appended, s_flag, s_level, s_span_lo,
      s_span_hi;
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const lg_guard_params &p = a.p;
  const lg_token_params &tp = a.tp;
  const int H = tp.hist, W = p.W;
  const int np = p.p_max - p.p_min + 1;
  int32_t *tok_s = sm;          // [H] token of position q at q % H
  int32_t *lm_s = sm + H;       // [H] latest earlier equal token of the window at arrival
  // the compression ratio's arrays: the window, each position's phrase end (two buffers for
  // the pointer jumping) and phrase count
  int32_t *x_s = sm + 2 * H;  // [W]
  auto nx_s = [&](int buf) { return x_s + (1 + buf) * W; };  // [W] each, buf 0 or 1
  auto ct_s = [&](int buf) { return x_s + (3 + buf) * W; };  // [W] each
  int32_t *ts = a.tstate + (int64_t)b * state_stride(H, np);
  int32_t *ring_tok = ts + kHdrWords, *ring_lm = ts + kHdrWords + H;
  int32_t *run = ts + kHdrWords + 2 * H;

  const int n = a.c.len[b];
  const int y = a.tokens[b];
  const double pm = (double)a.pmax[b];
  const int t = ts[0];  // tokens before this one: this token is position t
  const int synced = ts[2] - 1, app_old = ts[3];
  const int kc = a.kept_count ? a.kept_count[b] : -1;
  const int B = a.prune ? a.budget[b] : 0;
  int4 st_a = make_int4(0, 0, 0, 0), st_b = make_int4(0, 0, 0, 0);
  if (tid == 0) {
    st_a = reinterpret_cast<const int4 *>(a.state + b)[0];
    st_b = reinterpret_cast<const int4 *>(a.state + b)[1];
  }
  if (cta_status_bad(a.c.dev_status)) return;
  const int Tn = t + 1;
  for (int k = tid; k < H; k += kTokThreads) {
    tok_s[k] = ring_tok[k];
    lm_s[k] = ring_lm[k];
  }
  __syncthreads();
  if (tid == 0) tok_s[t % H] = y;
  __syncthreads();
  auto tok = [&](int q) { return tok_s[q % H]; };
  const int wlo = max(0, Tn - W);
  const int w = Tn - wlo;

  // (1) this token against the window (latest earlier equal token) and every period
  const int j0 = t - 1 - tid;
  bool m0 = false;
  int latest = -1;
  if (j0 >= 0 && j0 > t - H) {
    m0 = tok(j0) == y;
    if (m0 && j0 >= wlo) latest = j0;
  }
  if (latest < 0)
    for (int j = j0 - kTokThreads; j >= wlo; j -= kTokThreads)
      if (tok(j) == y) {
        latest = j;
        break;
      }
  int pstar = 0x7fffffff;
  for (int pi = tid; pi < np; pi += kTokThreads) {
    const int P = p.p_min + pi;
    const int cap = max(p.m_rep * P, p.l_min);
    const int j = t - P;
    const bool m = j >= 0 && (P == tid + 1 ? m0 : tok(j) == y);
    const int r = m ? min(run[pi] + 1, cap) : 0;
    run[pi] = r;
    if (pstar == 0x7fffffff && Tn >= cap + P && r >= cap) pstar = P;
  }
  // novel tokens of the window before this one
  int nov = 0, tail = 0;
  for (int q = wlo + tid; q < t; q += kTokThreads) {
    const int novel = lm_s[q % H] < wlo;
    nov += novel;
    if (q >= Tn - p.stall_len) tail += novel;
  }
  latest = __reduce_max_sync(0xffffffffu, latest);
  nov = __reduce_add_sync(0xffffffffu, nov);
  tail = __reduce_add_sync(0xffffffffu, tail);
  pstar = (int)__reduce_min_sync(0xffffffffu, (unsigned)pstar);
  // after a prune of this sequence: the kept rows that end the kept list one after another up
  // to the old last row, and were consecutive tokens before, still are (first break from the end)
  const bool use_kept = kc >= 0 && synced >= 0 && n == kc + 1;
  const int run_lim = use_kept ? min(kc, app_old) : 0;
  int first_bad = 0x7fffffff;
  if (use_kept) {
    const int32_t *K = a.kept_idx + (int64_t)b * a.max_keep;
    for (int jo = tid; jo < run_lim; jo += kTokThreads) {
      const int v = K[kc - 1 - jo];
      if (v != synced - 1 - jo || v < synced - app_old) {
        first_bad = jo;
        break;
      }
    }
  }
  first_bad = (int)__reduce_min_sync(0xffffffffu, (unsigned)first_bad);
  if (lane == 0) {
    w_latest[warp] = latest;
    w_nov[warp] = nov;
    w_tail[warp] = tail;
    w_pstar[warp] = pstar;
    w_run[warp] = first_bad;
  }

  // (2) compression ratio of the window, every cr_every tokens.  The greedy parse takes at
  // position i the longest earlier match (overlap allowed) when it is two tokens or more, else
  // one literal token.  The longest match at every i comes first, all at once: along each
  // diagonal d (an earlier start i - d) the run of equal pairs from i to the window's end,
  // scanned from the end, a lane per diagonal and the warp's maximum at each position; the
  // parse is then a chain of phrase ends from 0, whose length pointer jumping finds in
  // ceil(log2 w) rounds.
  const bool eval_cr = t % tp.cr_every == 0;
  int phrases = 0;
  if (eval_cr) {
    for (int k = tid; k < w; k += kTokThreads) {
      x_s[k] = tok(wlo + k);
      nx_s(0)[k] = 0;  // longest earlier match at k, kept only from two tokens on
    }
    __syncthreads();
    for (int d0 = 1 + warp * 32; d0 < w; d0 += kTokThreads) {
      const int d = d0 + lane;
      int r = 0;
      // 32-position blocks [base, top] from the end; the lane of position i keeps the warp's
      // maximum at i and writes it once per block
      for (int top = w - 1; top >= d0;) {
        const int base = max(top & ~31, d0);
        int acc = 0;
#pragma unroll 4
        for (int i = top; i >= base; --i) {
          r = (i >= d && x_s[i] == x_s[i - d]) ? r + 1 : 0;
          const int m = (int)__reduce_max_sync(0xffffffffu, (unsigned)r);
          acc = lane == (i & 31) ? m : acc;
        }
        const int pos = (top & ~31) + lane;
        if (pos >= base && pos <= top && acc >= 2) atomicMax(&nx_s(0)[pos], acc);
        top = base - 1;
      }
    }
    __syncthreads();
    for (int k = tid; k < w; k += kTokThreads) {
      nx_s(0)[k] = k + max(nx_s(0)[k], 1);  // the next phrase's start (w: none)
      ct_s(0)[k] = 1;
    }
    __syncthreads();
    int cur = 0;
    for (int span = 1; span < w; span *= 2) {
      for (int k = tid; k < w; k += kTokThreads) {
        const int nk = nx_s(cur)[k];
        const bool in = nk < w;
        nx_s(cur ^ 1)[k] = in ? nx_s(cur)[nk] : nk;
        ct_s(cur ^ 1)[k] = ct_s(cur)[k] + (in ? ct_s(cur)[nk] : 0);
      }
      __syncthreads();
      cur ^= 1;
    }
    phrases = ct_s(cur)[0];
  }
  __syncthreads();

  // (3) votes, gates, trigger, state (thread 0)
  if (tid == 0) {
    int lt = -1, nv = 0, tl = 0, ps = 0x7fffffff, fb = 0x7fffffff;
    for (int k = 0; k < kTokWarps; ++k) {
      lt = max(lt, w_latest[k]);
      nv += w_nov[k];
      tl += w_tail[k];
      ps = min(ps, w_pstar[k]);
      fb = min(fb, w_run[k]);
    }
    const int novel = lt < wlo;
    nv += novel;
    tl += p.stall_len >= 1 ? novel : 0;
    const double ttr = (double)nv / (double)w;
    double cr;
    if (eval_cr) {
      cr = (double)phrases / (double)w;
      reinterpret_cast<double *>(ts + 4)[0] = cr;
    } else {
      cr = reinterpret_cast<const double *>(ts + 4)[0];
    }
    const int streak = pm > tp.theta_conf ? ts[1] + 1 : 0;
    const int sig1 = ttr < p.theta_ttr;
    const int sig2 = cr < tp.theta_cr;
    const int sig3 = streak >= tp.theta_streak;
    const int warn = sig1 + sig2 + sig3 >= p.K;
    const int stall = w >= p.stall_len && p.stall_len > 0 &&
                      (double)tl / (double)p.stall_len < p.theta_nov;
    const int tailrep = ps != 0x7fffffff;
    const int trig = st_a.x >= p.t_min && st_a.y == 0 && warn && (stall || tailrep);
    int appended;
    if (use_kept)
      appended = min(fb, run_lim) + 1;
    else
      appended = (synced >= 0 && n == synced + 1) ? app_old + 1 : 1;
    appended = min(appended, n);
    if (a.diag) {
      double *dg = a.diag + 8 * b;
      dg[0] = ttr;
      dg[1] = cr;
      dg[2] = streak;
      dg[3] = sig1;
      dg[4] = sig2;
      dg[5] = sig3;
      dg[6] = stall;
      dg[7] = tailrep ? ps : 0;
    }
    ts[0] = Tn;
    ts[1] = streak;
    ts[2] = n + 1;
    ts[3] = appended;
    ring_tok[t % H] = y;
    ring_lm[t % H] = lt;
    // x = t_gen, y = cd, z = level, w = last_trig; st_b.x = n_int
    if (trig) {
      const bool quick = st_a.x - st_a.w <= p.retrig_window;
      st_a.z = quick ? min(st_a.z + 1, p.level_max) : 0;
      st_a.w = st_a.x;
      st_a.y = p.cooldown;
      st_b.x += 1;
    } else if (st_a.y > 0) {
      st_a.y -= 1;
    }
    st_a.x += 1;
    reinterpret_cast<int4 *>(a.state + b)[0] = st_a;
    reinterpret_cast<int4 *>(a.state + b)[1] = st_b;
    s_trig = trig && tailrep;
    s_P = ps;
    s_n_tok = Tn;
    s_appended = appended;
    s_mismatch = -1;
    s_flag = trig;
    s_level = st_a.z;
    s_span_lo = s_span_hi = 0;
    a.flags[b] = trig;
    a.spans[2 * b] = 0;
    a.spans[2 * b + 1] = 0;
  }
  __syncthreads();

  // (4) span: the verified run extended back while tokens keep equalling the token P* earlier
  if (s_trig) {
    const int P = s_P;
    const int span_len = max(p.m_rep * P, p.l_min);
    const int lo_ext = max(0, Tn - H) + P;
    int s = Tn - span_len;
    if (s > lo_ext) {
      for (int hi = s; hi > lo_ext; hi -= kTokThreads) {
        const int i = hi - 1 - tid;
        if (i >= lo_ext && tok(i) != tok(i - P)) atomicMax(&s_mismatch, i);
        __syncthreads();
        const int found = s_mismatch;
        __syncthreads();
        if (found >= 0) break;
      }
      s = s_mismatch >= 0 ? s_mismatch + 1 : lo_ext;
    }
    if (tid == 0) {
      const int bad = min(s_n_tok - (s - P), s_appended);
      a.spans[2 * b] = n - bad;
      a.spans[2 * b + 1] = n;
      s_span_lo = n - bad;
      s_span_hi = n;
    }
  }

  // (5) fused prune: the retained set of this sequence from the decision just taken, the span
  // clipped to W^recent by keep_plan as in lg_prune_compact.  Every read of the previous kept
  // lists (1) lies before the barrier of (3), so they may be overwritten now.
  if (a.prune) {
    __syncthreads();  // thread 0's span
    const int code = write_keep(a.c, b, n, B, s_flag, s_span_lo, s_span_hi, s_level, p,
                                a.kept_idx, a.kept_count, a.max_keep, a.max_len, tid,
                                kTokThreads);
    if (code && tid == 0) set_status(a.c.dev_status, code);
  }
}

}  // namespace

size_t token_state_words(const lg_guard_params &p, const lg_token_params &tp) {
  return (size_t)state_stride(tp.hist, p.p_max - p.p_min + 1);
}

size_t token_smem_bytes(const lg_guard_params &p, const lg_token_params &tp) {
  return (size_t)(2 * tp.hist + 5 * p.W) * 4;
}

cudaError_t launch_token_detect(const lg_cache &c, const int32_t *tokens, const float *pmax,
                                int32_t *kept_idx, int32_t *kept_count, int max_keep,
                                lg_guard_state *state, const lg_guard_params &p,
                                const lg_token_params &tp, int32_t *flags, int32_t *spans,
                                double *diag, void *tstate, const int32_t *budget, int max_len,
                                cudaStream_t s) {
  TokenArgs a;
  a.c = c;
  a.tokens = tokens;
  a.pmax = pmax;
  a.kept_idx = kept_idx;
  a.kept_count = kept_count;
  a.max_keep = max_keep;
  a.budget = budget;
  a.max_len = max_len;
  a.prune = budget != nullptr;
  a.state = state;
  a.p = p;
  a.tp = tp;
  a.flags = flags;
  a.spans = spans;
  a.diag = diag;
  a.tstate = (int32_t *)tstate;
  const size_t smem = token_smem_bytes(p, tp);
  cudaError_t e = cudaFuncSetAttribute(token_detect_kernel,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  LG_TRY(launch_pdl(token_detect_kernel, c.batch, kTokThreads, smem, s, a));
  return cudaGetLastError();
}

}  // namespace lg
