/*
 * lg.h -- C ABI of the LoopGuard decode-path library (liblg.so), GB300 / sm_103a.
 *
 * LoopGuard (arXiv 2604.10044) guards long-context decoding against repetition loops: each
 * decode step attends over the KV cache (Sec. 3.1, Eq. 1), runs an online loop-onset test
 * (Sec. 5.2, Eq. 8, Eq. 9) and, when it fires or the cache is over its budget B, keeps the
 * retained set I_keep = anchors + sparse long-range rows + tail-cleaned recent rows
 * (Sec. 5.3, Eq. 10, Eq. 11) by an index-gather over every layer and kv-head.  An H2O
 * heavy-hitter eviction path (Sec. 2.2, Sec. 6.1) is the comparator policy.
 *
 * A decode step on this ABI:
 *   lg_begin_step -> lg_append -> lg_decode_attend -> lg_detect -> lg_prune_compact
 *   (lg_detect_prune fuses the last two), or with the token-level monitor:
 *   lg_begin_step -> lg_append -> lg_decode_attend -> lg_token_detect -> lg_prune_compact
 *   (lg_token_detect_prune fuses the last two)
 * or, on the comparator path:
 *   lg_begin_step -> lg_append -> lg_decode_attend(accumulate_h2o=1) -> lg_h2o_evict
 *
 * Conventions
 *  - Every pointer inside lg_cache and every array argument marked "device" is device memory
 *    owned by the caller; the library allocates nothing and keeps no global state, except
 *    the static scratch array that lg_decode_attend_noalloc uses in place of a workspace and
 *    two lookups cached for the process (the driver's tensor-map encoder, and per GPU the
 *    compaction kernel's resident CTAs), which no result depends on.
 *  - Every call is asynchronous on the caller's stream; nothing synchronises except
 *    lg_read_device_status.
 *  - Kernels are launched with programmatic stream serialization (programmatic dependent
 *    launch): each may be scheduled while the kernel before it in the stream is still running,
 *    and waits (griddepcontrol.wait) for that kernel to complete before it touches memory, so
 *    stream order holds as usual.  One exception, invisible to the caller: lg_detect's kernel
 *    reads the lengths, the monitor state and the sketches before its wait, then reads the
 *    length, the synced length and the new row again after it and drops everything read early
 *    unless all three are unchanged.  Only a library kernel can be running at that point: a
 *    kernel of the caller's (launched without the attribute) completes before the next
 *    kernel starts.  A kernel of the caller's that follows one of the library's on the same
 *    stream keeps full stream order unless the caller launches it with the same attribute, in
 *    which case it must wait the same way.
 *  - Arguments are validated on the host before any launch (null or misaligned pointers,
 *    unsupported shapes, short workspaces): the call returns an error and launches nothing.
 *  - Errors only visible on the device (a length above its capacity or above the call's
 *    max_len, a budget too small for the anchors, a bounded wait that ran out) are written
 *    once to *dev_status (first error wins) and every later kernel on that cache skips its
 *    work while the status is non-zero.  No kernel traps or asserts.
 *  - Shapes: head_dim d in {64, 128}; dtype bf16 or fp32; GQA group g = H_q / H_kv in 1..8.
 */
#ifndef LG_H
#define LG_H

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime.h>

#if defined(__GNUC__)
#define LG_API __attribute__((visibility("default")))
#else
#define LG_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  LG_OK = 0,
  LG_ERR_INVALID_ARG = 1, /* null/misaligned pointer, bad shape or range        */
  LG_ERR_UNSUPPORTED = 2, /* head_dim, dtype or GQA group not supported        */
  LG_ERR_CUDA = 3,        /* a CUDA launch failed                               */
  LG_ERR_CAPACITY = 4,    /* device: a sequence ran out of slots, or max_len
                             smaller than a current length                      */
  LG_ERR_TIMEOUT = 5,     /* device: a bounded wait on a copy ran out          */
  LG_ERR_WORKSPACE = 6,   /* workspace missing or smaller than required        */
  LG_ERR_BUDGET = 7       /* device: a budget leaves no room for the retained set */
} lg_status;

typedef enum { LG_BF16 = 0, LG_F32 = 1 } lg_dtype;

/* The KV cache of a batch of sequences (Sec. 3.1).  Row i of sequence b, layer l, kv-head h
   lives at slot seq_off[b] + i of the [L][H_kv][S_total][d] arrays; slots [0, len[b]) are the
   retained set S_t in ascending token order (on the H2O path, in slot order with pos[]
   holding each slot's token position). */
typedef struct {
  void *k;               /* device [L][H_kv][S_total][d], dtype; 16-byte aligned          */
  void *v;               /* device [L][H_kv][S_total][d], dtype; 16-byte aligned          */
  int32_t dtype;         /* lg_dtype                                                      */
  int32_t L, H_kv, d;    /* layers, kv-heads, head_dim                                    */
  int32_t batch;         /* sequences                                                     */
  int32_t pad;
  int64_t S_total;       /* slots per (layer, kv-head)                                    */
  const int64_t *seq_off;/* device [batch] first slot of each sequence                    */
  const int32_t *cap;    /* device [batch] slots owned by each sequence                   */
  int32_t *len;          /* device [batch] rows in use (updated by the calls)             */
  uint32_t *sketch;      /* device [S_total][H_kv*d/32] sign bits of the guard layer's
                            V rows (bit j of word w = sign bit of element 32w+j of the
                            row flattened as [H_kv][d]); nullable on the H2O path        */
  float *h2o;            /* device [L][H_kv][S_total] accumulated attention, H2O path;
                            nullable                                                      */
  int32_t *pos;          /* device [L][H_kv][S_total] token position of each slot, H2O
                            path; nullable                                                */
  int32_t *dev_status;   /* device [1] sticky error code, 0 = ok                          */
} lg_cache;

/* Per-sequence guard state (Sec. 5.2, Sec. 5.3): 32 bytes, device resident, plain bytes that
   can be saved and restored with the cache. */
typedef struct {
  int32_t t_gen;     /* decode steps seen (warmup: Trigger needs t_gen >= t_min, Eq. 9) */
  int32_t cd;        /* cooldown counter cd(t) (Eq. 9)                                   */
  int32_t level;     /* aggressiveness level l of the recent budget (Sec. 5.3)           */
  int32_t last_trig; /* t_gen of the last intervention                                   */
  int32_t n_int;     /* interventions so far                                             */
  int32_t pad[3];
} lg_guard_state;

/* Guard hyper-parameters.  Paper values: W = 256, K = 2, N_anchor = 32 (Sec. 6.1),
   theta_ttr = 0.2, theta_nov = 0.02, theta_stall = 4, t_min = 64, cooldown 32 (App. B.2).
   The paper detects on generated tokens; this library restates each signal over attention
   statistics and V-row sketches, and the remaining fields are that restatement's constants
   (defaults from lg_default_params). */
typedef struct {
  int32_t W;             /* monitor window, rows                                         */
  int32_t K;             /* votes needed out of 3 (Eq. 8)                                */
  int32_t t_min;         /* warmup (Eq. 9)                                               */
  int32_t cooldown;      /* steps blocked after an intervention                         */
  int32_t n_anchor;      /* anchor prefix kept by every prune (Sec. 5.3)                 */
  int32_t stall_len;     /* theta_stall: rows of the novelty-stagnation gate             */
  int32_t p_min, p_max;  /* period search range of the tail self-alignment test          */
  int32_t l_min;         /* minimum verified tail length                                 */
  int32_t m_rep;         /* verified tail covers m_rep periods (the debounce)            */
  int32_t suffix_w;      /* W_s: rows of the suffix-mass statistic                       */
  int32_t guard_layer;   /* layer whose V rows are sketched                              */
  int32_t level_max;     /* cap of the aggressiveness level                              */
  int32_t retrig_window; /* re-trigger within this many steps raises the level           */
  int32_t headroom;      /* rows freed below B by a prune: min(headroom, B/4)            */
  int32_t pad;
  double theta_ttr;      /* vote 1: novel-row fraction of the window below this          */
  double theta_nov;      /* stall: novel fraction of the last stall_len rows below this  */
  double theta_ent;      /* vote 2: mean normalised attention entropy below this         */
  double theta_lift;     /* vote 3: mean suffix lift S*n/W_s at or above this            */
  double tau_ham;        /* rows match when Hamming distance <= floor(tau_ham * bits)    */
} lg_guard_params;

/* Fills *p with the defaults listed above (paper values where the paper gives one). */
LG_API lg_status lg_default_params(lg_guard_params *p);

/* Human-readable name of a status code; never NULL. */
LG_API const char *lg_status_string(lg_status s);

/* Workspace bytes lg_decode_attend needs for n_layers layers at lengths <= max_len
   (split-K partials, plus logits when accumulate_h2o). */
LG_API size_t lg_workspace_size(const lg_cache *c, int H_q, int n_layers, int max_len,
                         int accumulate_h2o);

/* Sets state[b] = {t_gen0, 0, 0, never, 0} for every sequence (device array [batch]). */
LG_API lg_status lg_state_init(const lg_cache *c, lg_guard_state *state, int t_gen0, cudaStream_t s);

/* Reserves this step's slot: len[b] += 1 for every sequence.  A sequence whose len equals its
   cap sets LG_ERR_CAPACITY on the device and keeps its length. */
LG_API lg_status lg_begin_step(const lg_cache *c, cudaStream_t s);

/* Appends the step's K/V rows (Sec. 3.1: the new token's key and value join the cache) at
   slot len[b]-1 of layers [layer0, layer0+n_layers).
   k_new, v_new: device [n_layers][batch][H_kv][d], dtype, 16-byte aligned.
   pos_new: device [batch] token position of the new row, required when c->pos is set (the
   row's H2O score is reset to 0 there).  When p->guard_layer is in the range, the row's
   sketch is written too.  Call after lg_begin_step. */
LG_API lg_status lg_append(const lg_cache *c, int layer0, int n_layers, const void *k_new,
                    const void *v_new, const int32_t *pos_new, const lg_guard_params *p,
                    cudaStream_t s);

/* Sketches of the guard layer's rows [0, len[b]) of every sequence (after a prefill). */
LG_API lg_status lg_sketch_build(const lg_cache *c, const lg_guard_params *p, int max_len,
                          cudaStream_t s);

/* Decode attention over the retained set (Sec. 3.1, Eq. 1) for layers [layer0,
   layer0+n_layers), fused with the per-head statistics the guard reads:
     out[l][b][h][:] = sum_i a_i v_i,  a = softmax_i(<q, k_i> * scale) over i < len[b]
     stats[l][b][h] = {m, l, H, S}: m = max_i s_i, l = sum_i exp(s_i - m),
                      H = -sum_i a_i ln a_i (nats), S = sum of a_i over the last
                      min(suffix_w, len[b]) rows
   q: device [n_layers][batch][H_q][d] dtype; out: device same shape, dtype;
   stats: device [n_layers][batch][H_q][4] fp32.  Query head h reads kv-head h / (H_q/H_kv).
   accumulate_h2o: also add sum over the GQA group of a_i to h2o[l][kvh][slot] (c->h2o).
   max_len: host bound on every len[b] (sizes the grid; a longer sequence is an error).
   ws: device workspace of at least lg_workspace_size(...) bytes, 256-byte aligned.  On the bf16
   path successive calls with one workspace walk the cache in alternating directions (one word
   of ws keeps the direction), so that a call starts on the rows the previous call read last,
   which may still be in L2; no result depends on the direction. */
LG_API lg_status lg_decode_attend(const lg_cache *c, int layer0, int n_layers, const void *q, int H_q,
                           float scale, void *out, float *stats, int suffix_w,
                           int accumulate_h2o, int max_len, void *ws, size_t ws_bytes,
                           cudaStream_t s);

/* Online loop-onset test (Sec. 5.2, Eq. 8, Eq. 9), one pass per sequence:
     vote 1 (diversity, restating m_ttr < theta_ttr): novel rows of the last min(W, n)
       sketches / window < theta_ttr; a row is novel when no earlier row of the window
       matches it;
     vote 2 (confidence collapse, restated): mean over layers and heads of H / ln n below
       theta_ent;
     vote 3 (redundancy / locking, restated): mean of S * n / W_s at or above theta_lift;
     Warn = votes >= K; Stall = novel fraction of the last stall_len rows < theta_nov;
     TailRep = some P in [p_min, p_max] with each of the last max(m_rep P, l_min) rows
       matching the row P earlier (smallest such P is P*);
     Trigger = t_gen >= t_min and cd = 0 and Warn and (Stall or TailRep).
   On a trigger with TailRep the span [lo, hi) of I_bad covers every copy of the period
   extended back while rows keep matching, clipped to W^recent = [n - budget/2, n).
   stats: device [L][batch][H_q][4], 16-byte aligned (lg_decode_attend's output for all
   layers); state: device [batch], 16-byte aligned; budget: device [batch]; flags: device
   [batch] (1 = trigger);
   spans: device [batch][2] ([0,0) when empty).
   diag: nullable device [batch][8] fp64, per sequence {mean normalised entropy, mean suffix
   lift, novel fraction, vote 1, vote 2, vote 3, Stall, P* (0 = no tail repetition)}.  Each
   vote is the fp64 quotient's decision against its threshold (the kernel compares counts and
   fixed-point sums with bounds and divides only next to a threshold).
   dstate: device, lg_detect_state_size bytes, zero-filled before the first call on a cache and
   after any change of W or of the period range.  It carries the monitor from call to call (for
   each slot the latest earlier matching row, for each period the trailing matching run), so a
   step that appended one row costs O(W + p_max - p_min) row comparisons (Sec. 5.4); after a
   prune, or any other change of a length, the call recomputes it from the sketches. */
LG_API lg_status lg_detect(const lg_cache *c, const float *stats, int H_q, lg_guard_state *state,
                           const int32_t *budget, const lg_guard_params *p, int32_t *flags,
                           int32_t *spans, double *diag, void *dstate, cudaStream_t s);

/* Parameters of the token-level monitor (lg_token_detect). */
typedef struct {
  int32_t cr_every;      /* the compression ratio is evaluated every cr_every tokens      */
  int32_t theta_streak;  /* confidence-collapse streak, steps (App. B.2: 6)                */
  int32_t hist;          /* generated tokens kept per sequence (>= W and >= p_max +
                            max(m_rep p_max, l_min)); the span reaches back at most as far */
  int32_t pad;
  double theta_cr;       /* redundancy threshold (App. B.2: 0.12)                           */
  double theta_conf;     /* top-1 probability threshold (App. B.2: 0.9)                     */
} lg_token_params;

/* Fills *tp with the defaults: cr_every 16, theta_streak 6, hist 512, theta_cr 0.12,
   theta_conf 0.9. */
LG_API lg_status lg_default_token_params(lg_token_params *tp);

/* Bytes of lg_token_detect's tstate: batch times (16 + 2 hist + p_max - p_min + 1) 32-bit
   words rounded up to a multiple of 4; 0 on invalid arguments. */
LG_API size_t lg_token_state_size(const lg_cache *c, const lg_guard_params *p,
                                  const lg_token_params *tp);

/* Token-level loop-onset monitor (Sec. 5.2, Eq. 8, Eq. 9, App. B.2; indicators of Sec. 4.3),
   one step per call, for callers that have the generated token ids and top-1 probabilities:
     window W_t = the last min(W, t) generated tokens; a token of W_t is novel when no earlier
       token of W_t equals it;
     vote 1: novel tokens / |W_t| (TTR) < theta_ttr;
     vote 2: greedy LZ77 phrases of W_t / |W_t| (CR; a phrase is the longest earlier match of
       >= 2 tokens, overlap allowed, else one literal token), evaluated every cr_every tokens
       and held in between, < theta_cr;
     vote 3: consecutive steps with p_max > theta_conf >= theta_streak;
     Stall: novel fraction of the last stall_len tokens < theta_nov;
     TailRep: smallest P in [p_min, p_max] whose last max(m_rep P, l_min) tokens each equal
       the token P earlier (P*);
     Trigger = t_gen >= t_min and cd = 0 and votes >= K and (Stall or TailRep).
   On a trigger with TailRep the span [lo, hi) covers the verified run extended back while
   tokens keep equalling the token P* earlier (at most hist tokens back) plus its first period,
   mapped onto the trailing cache rows that hold consecutive generated tokens (hi = len[b]):
   the rows appended one per step since the cache last changed otherwise, or, when the caller
   passes the retained lists of the prune that followed the previous call, also the kept rows
   that end the kept list one after another up to the old last row (a budget cut keeps its
   recent rows so).  The span is not clipped here: lg_prune_compact, which takes
   flags, spans and state as from lg_detect, clips it to W^recent.
   tokens: device [batch] int32, this step's generated token; pmax: device [batch] fp32.
   kept_idx, kept_count, max_keep: nullable (both or neither): the kept_idx/kept_count buffers
   lg_prune_compact wrote after the previous call (kept_count -1 = not pruned), as laid out
   there.  state (16-byte aligned), flags, spans as for lg_detect; diag: nullable device [batch][8]
   fp64 {TTR, CR, streak, vote 1, vote 2, vote 3, Stall, P* (0 = none)}.
   tstate: device, lg_token_state_size bytes, 8-byte aligned, zero-filled before the first
   call.  Call it once per decode step after the step's append (len[b] counts this step's
   row). */
LG_API lg_status lg_token_detect(const lg_cache *c, const int32_t *tokens, const float *pmax,
                                 const int32_t *kept_idx, const int32_t *kept_count,
                                 int max_keep, lg_guard_state *state, const lg_guard_params *p,
                                 const lg_token_params *tp, int32_t *flags, int32_t *spans,
                                 double *diag, void *tstate, cudaStream_t s);

/* lg_token_detect (passed the kept lists) followed by lg_prune_compact (same results, same
   device state), with the retained set formed by the token-level monitor's own kernel: two
   kernel launches instead of three.  kept_idx and kept_count are required: the kernel reads
   the previous prune's lists from them (as lg_token_detect does) and then writes this step's
   over them (as lg_prune_compact does).  budget, max_keep and max_len as for lg_prune_compact;
   validation is the union of both calls'. */
LG_API lg_status lg_token_detect_prune(const lg_cache *c, const int32_t *tokens,
                                       const float *pmax, lg_guard_state *state,
                                       const int32_t *budget, const lg_guard_params *p,
                                       const lg_token_params *tp, int32_t *flags, int32_t *spans,
                                       double *diag, void *tstate, int32_t *kept_idx,
                                       int32_t *kept_count, int max_keep, int max_len,
                                       cudaStream_t s);

/* Bytes of lg_detect's dstate: (batch * (p_max - p_min + 3) + S_total) 32-bit words. */
LG_API size_t lg_detect_state_size(const lg_cache *c, const lg_guard_params *p);

/* Retained set and in-place index-gather (Sec. 5.3, Eq. 10, Eq. 11) for every sequence with
   flags[b] = 1 or len[b] > budget[b]:
     I_keep = [0, N_anchor) + a uniform lattice of B_sparse rows over [N_anchor, n - R)
              + the last B_recent(level) rows of [n - R, n) outside the span,
     R = B/2, B_recent(l) = (B/4) >> l, B_sparse = B - min(headroom, B/4) - N_anchor - B/4;
   a budget event without a trigger uses level 0 and no span.  Rows of K, V (every layer and
   kv-head) and the sketches move to slots 0..|I_keep|-1 in order; len[b] = |I_keep|.
   kept_idx: device [batch][max_keep] ascending slot lists; kept_count: device [batch]
   (|I_keep|, or -1 for a sequence left as it was).  max_keep >= every budget[b].
   max_len: host bound on every len[b]. */
LG_API lg_status lg_prune_compact(const lg_cache *c, const int32_t *flags, const int32_t *spans,
                           const lg_guard_state *state, const int32_t *budget,
                           const lg_guard_params *p, int32_t *kept_idx, int32_t *kept_count,
                           int max_keep, int max_len, cudaStream_t s);

/* lg_detect followed by lg_prune_compact (same arguments, same results, same device state),
   with the retained set formed by the loop-onset test's own kernel: two kernel launches instead
   of three.  Validation is the union of both calls'; dstate and the kept lists as there. */
LG_API lg_status lg_detect_prune(const lg_cache *c, const float *stats, int H_q,
                                 lg_guard_state *state, const int32_t *budget,
                                 const lg_guard_params *p, int32_t *flags, int32_t *spans,
                                 double *diag, void *dstate, int32_t *kept_idx,
                                 int32_t *kept_count, int max_keep, int max_len, cudaStream_t s);

/* H2O comparator state: pos[l][h][slot] = slot and h2o = 0 for slots [0, len[b]) (after a
   prefill whose rows are in token order). */
LG_API lg_status lg_h2o_reset(const lg_cache *c, int max_len, cudaStream_t s);

/* H2O comparator eviction (heavy hitters by accumulated attention, Sec. 2.2, Sec. 6.1) for
   every sequence with len[b] > budget[b], independently per (layer, kv-head):
     recent rows (pos > pos_now[b] - budget[b]/2) are kept; of the others the highest
     (score, pos) are kept up to budget[b] rows in total;
     len[b] = budget[b] + 1: the one evicted slot is refilled from slot len-1;
     otherwise: the kept rows move to slots 0..budget-1 in order.
   pos_now: device [batch] position of the newest token. */
LG_API lg_status lg_h2o_evict(const lg_cache *c, const int32_t *budget, const int32_t *pos_now,
                       int max_len, cudaStream_t s);

/* Maximum scratch of lg_decode_attend_noalloc: 32 MiB of device memory per GPU. */
#define LG_NOALLOC_SCRATCH_BYTES (32u << 20)

/* lg_decode_attend for callers that cannot allocate device memory (a plugin inside a framework
   that owns every device allocation, or a latency-critical loop that cannot take cudaMalloc's
   implicit synchronisation).  The paper has no counterpart; this is a deployment variant.
   Same arguments and results as lg_decode_attend, without ws / ws_bytes: the scratch is a
   statically sized array of this library (LG_NOALLOC_SCRATCH_BYTES per GPU that loads the
   library, held until the process exits), and the call allocates nothing.
   - A call whose workspace (lg_workspace_size) exceeds LG_NOALLOC_SCRATCH_BYTES returns
     LG_ERR_WORKSPACE and launches nothing.
   - The first call on each device looks up the array's device address (cudaGetSymbolAddress,
     with that device current); make that first call before any stream capture.
   - Every call on a device shares the one array, and it keeps the last call's contents (no
     clearing is needed: every scratch byte read is written earlier in the same call, except
     one word whose low bit picks the direction in which the call walks the cache, which never
     changes a result).  Calls that overlap on the GPU (different streams without ordering)
     race on it: order them. */
LG_API lg_status lg_decode_attend_noalloc(const lg_cache *c, int layer0, int n_layers,
                                          const void *q, int H_q, float scale, void *out,
                                          float *stats, int suffix_w, int accumulate_h2o,
                                          int max_len, cudaStream_t s);

/* StreamingLLM comparator eviction (attention sinks + sliding window, Sec. 2.2, Sec. 6.1) for
   every sequence with len[b] > budget[b], per (layer, kv-head): positions < n_sink and the
   budget[b] - n_sink newest positions stay.  len[b] = budget[b] + 1: the oldest non-sink slot
   is refilled from slot len-1; otherwise the kept rows move to slots 0..budget-1 in order.
   Uses c->pos (positions are written by lg_append; lg_h2o_reset initialises them). */
LG_API lg_status lg_streaming_evict(const lg_cache *c, const int32_t *budget,
                                    const int32_t *pos_now, int n_sink, int max_len,
                                    cudaStream_t s);

/* Copies *dev_status to *host_code after synchronising the stream. */
LG_API lg_status lg_read_device_status(const lg_cache *c, int32_t *host_code, cudaStream_t s);

#ifdef __cplusplus
}
#endif
#endif
