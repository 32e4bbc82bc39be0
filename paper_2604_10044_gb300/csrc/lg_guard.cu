// Cache bookkeeping, the loop-onset test, the retained-set construction with its in-place
// index-gather, and the H2O comparator eviction (LoopGuard Sec. 5.2, Sec. 5.3; H2O Sec. 2.2,
// Sec. 6.1).
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <limits.h>
#include <math.h>
#include <stdint.h>

#include <atomic>

#include "lg_common.cuh"
#include "lg_internal.h"
#include "lg_keep.cuh"
#include "lg_votes.cuh"

namespace lg {

// ------------------------------------------------------------------ step bookkeeping

// (Here and in append_kernel the inputs are read before the status word, so that every load
// of a thread is in flight at once; neither kernel has a barrier after its status check.)
__global__ void begin_step_kernel(lg_cache c) {
  pdl_enter();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= c.batch) return;
  const int n = c.len[b], cap = c.cap[b];
  if (status_bad(c.dev_status)) return;
  if (n + 1 > cap)
    set_status(c.dev_status, LG_ERR_CAPACITY);
  else
    c.len[b] = n + 1;
}

// sketch word w of a row: sign bits of elements [32w, 32w+32) of the row flattened [H_kv][d]
template <typename T>
__device__ __forceinline__ uint32_t sketch_word(const void *row_base, int64_t head_stride, int d,
                                                int w) {
  uint32_t bits = 0;
#pragma unroll 4
  for (int j = 0; j < 32; ++j) {
    const int e = w * 32 + j;
    const int h = e / d, x = e % d;
    bits |= Elem<T>::sign(row_base, (int64_t)h * head_stride + x) << j;
  }
  return bits;
}

// Blocks [0, row_blocks): one thread per 16-byte chunk of a new row, written to slot
// len[b] - 1.  Blocks [row_blocks, row_blocks + batch) when the guard layer is in the call:
// the sketch of that layer's new V row (read from v_new [n_layers][b][H_kv][d]), a warp per
// word: lane j reads element 32w + j and the ballot of the sign bits is word w.
template <typename T>
__global__ void append_kernel(lg_cache c, int layer0, int n_layers, const uint4 *k_new,
                              const uint4 *v_new, const int32_t *pos_new, int row_blocks,
                              int lguard) {
  pdl_enter();
  if ((int)blockIdx.x >= row_blocks) {
    const int b = blockIdx.x - row_blocks;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nwords = c.H_kv * c.d / 32;
    const T *row = (const T *)v_new + ((int64_t)lguard * c.batch + b) * c.H_kv * c.d;
    // the sign bits this warp packs are requested with the length and the status (one round
    // trip for all), up to 8 words a warp at once
    constexpr int kWordsPerWarp = 8;
    const int wstep = blockDim.x >> 5;
    uint32_t sg[kWordsPerWarp];
#pragma unroll
    for (int k = 0; k < kWordsPerWarp; ++k) {
      const int w = warp + k * wstep;
      sg[k] = w < nwords ? Elem<T>::sign(row, w * 32 + lane) : 0u;
    }
    const int slot = c.len[b] - 1;
    const int64_t off = c.seq_off[b];
    // one status read per warp, so that every lane of the ballot takes the same branch
    const int bad = __shfl_sync(0xffffffffu, lane == 0 ? (int)status_bad(c.dev_status) : 0, 0);
    if (bad || slot < 0) return;
#pragma unroll
    for (int k = 0; k < kWordsPerWarp; ++k) {
      const int w = warp + k * wstep;
      const uint32_t word = __ballot_sync(0xffffffffu, sg[k] != 0u);
      if (lane == 0 && w < nwords) c.sketch[(off + slot) * nwords + w] = word;
    }
    for (int w = warp + kWordsPerWarp * wstep; w < nwords; w += wstep) {
      const uint32_t word = __ballot_sync(0xffffffffu, Elem<T>::sign(row, w * 32 + lane) != 0u);
      if (lane == 0) c.sketch[(off + slot) * nwords + w] = word;
    }
    return;
  }
  const int cpr = c.d * (int)sizeof(T) / 16;
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t rows = (int64_t)n_layers * c.batch * c.H_kv;
  if (t >= rows * cpr) return;
  const int64_t row = t / cpr;
  const int ch = (int)(t % cpr);
  const int kvh = (int)(row % c.H_kv);
  const int b = (int)((row / c.H_kv) % c.batch);
  const int layer = layer0 + (int)(row / ((int64_t)c.H_kv * c.batch));
  const uint4 kr = k_new[row * cpr + ch], vr = v_new[row * cpr + ch];
  const int slot = c.len[b] - 1;
  const int64_t off = c.seq_off[b];
  if (status_bad(c.dev_status)) return;
  if (slot < 0) {
    set_status(c.dev_status, LG_ERR_CAPACITY);
    return;
  }
  const int64_t s = ((int64_t)layer * c.H_kv + kvh) * c.S_total + off + slot;
  reinterpret_cast<uint4 *>(c.k)[s * cpr + ch] = kr;
  reinterpret_cast<uint4 *>(c.v)[s * cpr + ch] = vr;
  if (ch == 0 && c.pos) {
    c.pos[s] = pos_new[b];
    c.h2o[s] = 0.f;
  }
}

// sketches of rows [0, len[b]) of the guard layer, read from the cache
template <typename T>
__global__ void sketch_build_kernel(lg_cache c, int guard_layer, int max_len) {
  // no early start of the kernel after this one: the detect kernel reads sketch rows before its
  // dependency wait and checks only the length, its synced length and the newest row, which this
  // kernel leaves unchanged while it may rewrite every other row
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int b = blockIdx.y;
  if (status_bad(c.dev_status)) return;
  const int n = c.len[b];
  if (n > max_len) {
    if (threadIdx.x == 0 && blockIdx.x == 0) set_status(c.dev_status, LG_ERR_CAPACITY);
    return;
  }
  const int nwords = c.H_kv * c.d / 32;
  const int64_t total = (int64_t)n * nwords;
  const T *base = (const T *)c.v + ((int64_t)guard_layer * c.H_kv * c.S_total + c.seq_off[b]) * c.d;
  for (int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; t < total;
       t += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = t / nwords;
    const int w = (int)(t % nwords);
    c.sketch[(c.seq_off[b] + i) * nwords + w] =
        sketch_word<T>(base + i * c.d, c.S_total * c.d, c.d, w);
  }
}

__global__ void state_init_kernel(int batch, lg_guard_state *state, int t_gen0) {
  pdl_enter();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= batch) return;
  lg_guard_state s;
  s.t_gen = t_gen0;
  s.cd = 0;
  s.level = 0;
  s.last_trig = -(1 << 30);
  s.n_int = 0;
  s.pad[0] = s.pad[1] = s.pad[2] = 0;
  state[b] = s;
}

// ------------------------------------------------------------------ loop-onset test

struct DetectArgs {
  lg_cache c;
  const float *stats;  // [L][batch][H_q][4]
  int H_q;
  lg_guard_state *state;
  const int32_t *budget;
  lg_guard_params p;
  int32_t *flags, *spans;
  double *diag;
  int32_t *dstate;
  int nwords, thr, smem_rows;
  // nullable: when set, the same CTA goes on to the retained set (see write_keep)
  int32_t *kept_idx, *kept_count;
  int max_keep, max_len;
};

constexpr int kDetectThreads = 512;

// Hamming distance of two sketch rows <= thr, stopping once it is exceeded
__device__ __forceinline__ bool rows_match(const uint32_t *x, const uint32_t *y, int nwords,
                                           int thr) {
  int dist = 0;
  int w = 0;
  for (; w + 4 <= nwords; w += 4) {
    dist += __popc(x[w] ^ y[w]) + __popc(x[w + 1] ^ y[w + 1]) + __popc(x[w + 2] ^ y[w + 2]) +
            __popc(x[w + 3] ^ y[w + 3]);
    if (dist > thr) return false;
  }
  for (; w < nwords; ++w) dist += __popc(x[w] ^ y[w]);
  return dist <= thr;
}

// Full Hamming distance of two sketch rows of nwords words (nwords a multiple of 4, rows
// 16-byte aligned); the loads are independent, so a thread has all of them in flight at once,
// and go to L2 only (the detect kernel also calls this before its dependency wait, see below).
__device__ __forceinline__ int hamming(const uint32_t *x, const uint32_t *y, int nwords) {
  const uint4 *a = reinterpret_cast<const uint4 *>(x);
  const uint4 *b = reinterpret_cast<const uint4 *>(y);
  int dist = 0;
#pragma unroll 8
  for (int w = 0; w < nwords / 4; ++w) {
    const uint4 u = __ldcg(a + w), v = __ldcg(b + w);
    dist += __popc(u.x ^ v.x) + __popc(u.y ^ v.y) + __popc(u.z ^ v.z) + __popc(u.w ^ v.w);
  }
  return dist;
}

constexpr int kDetectWarps = kDetectThreads / 32;
constexpr int kStatWarps = 3;  // warps that sum the statistics (one per SM sub-partition)
constexpr int kStatBatch = 8;  // statistics loads a thread has in flight at once
constexpr float kFixScale = 1099511627776.0f;  // 2^40: statistics summed in 2^-40 units
constexpr int kCmpWarp0 = kStatWarps + 1;  // the new-row comparisons: warps after ln n's
constexpr int kCmpThreads = kDetectThreads - kCmpWarp0 * 32;
constexpr int kCmpBatch = 6;  // comparison chunks a thread has in flight at once
constexpr int kPreRowChunks = 64;  // sketch rows up to 1 KB (H_kv d <= 8192) take the early phase
static_assert(kCmpThreads % 32 == 0, "comparing threads in whole warps");

// One CTA per sequence, monitor state carried from call to call in dstate:
//   lm[slot]  latest earlier row of the window (as it was when the row was examined) whose
//             sketch matches the row, -1 if none.  Row i of the window [wlo, n) is novel iff
//             lm[i] < wlo, and this stays true as the window start moves forward.
//   run[P]    trailing rows (up to the test length) that match the row P earlier.
//   synced    the length seen by the previous call.
// When the length grew by exactly one row since the previous call, only the new row i = n-1 is
// examined, and before the kernel waits for the one before it (the attention pass, whose
// statistics it needs): the warps after the statistics warps compare the new row with every row
// the window and the periods need (the window comparisons double as the period comparisons), a
// row's 16-byte chunks on consecutive lanes, the distances in shared memory; then thread t takes
// window row i-1-t (and i-1-t-T, ...) for the latest match and period P = t+1's run, and every
// warp reduces its share (latest match, novel rows, shortest verified period), kept in shared
// memory; the ln n warp forms the votes' bounds.  After the wait three warps sum the statistics
// in 64-bit fixed point while the fourth checks that the early phase's inputs did not change;
// the early results are committed (or dropped for a recompute), and thread 0 takes the votes
// against the bounds (a division only next to a threshold) and updates the guard state.  At one
// sequence the CTA starts on an SM freed by the attention pass's first finishing CTAs, so the
// comparisons run beside the pass's last chunks and merges.  Otherwise (first call, after a
// prune or any other change of the cache) the window and the runs are recomputed after the
// wait: the sketches of the last smem_rows rows are staged in shared memory with a row stride
// of nwords + 1 words (rows that different lanes read fall in different banks), one warp scans
// each window row, one warp each period.
__global__ void __launch_bounds__(kDetectThreads, 1) detect_kernel(DetectArgs a) {
  extern __shared__ __align__(16) uint32_t sk_s[];
  __shared__ long long red_e[kStatWarps], red_l[kStatWarps];  // fixed point, 2^-40 units
  __shared__ int red_ok[kStatWarps];                          // every statistic finite
  __shared__ int w_latest[kDetectWarps], w_nov[kDetectWarps], w_nov_tail[kDetectWarps],
      w_pstar[kDetectWarps];
  __shared__ double s_logn;
  __shared__ FixBound s_bound_ent, s_bound_lift;  // sum-vote bounds, 2^-40 units, see (1)
  __shared__ int2 s_bound_ttr, s_bound_stall;       // count-vote bounds
  __shared__ int s_novel, s_novel_tail, s_pstar, s_mismatch, s_trig, s_span_lo, s_span_hi,
      s_level, s_bad, s_valid, s_latest, s_n0, s_synced0, s_n;
  __shared__ uint4 s_newrow[kPreRowChunks];  // the new sketch row as the early phase read it
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int32_t *status = a.c.dev_status;
  const int64_t off = a.c.seq_off[b];  // set by the caller, never written by a kernel
  const lg_guard_params &p = a.p;
  const int np = p.p_max - p.p_min + 1;
  int32_t *ds = a.dstate + (int64_t)b * (np + 2);
  const int nw = a.nwords, thr = a.thr, stride = nw + 1;
  const int cpr = nw / 4;  // 16-byte chunks per sketch row
  const uint32_t *sk_g = a.c.sketch + off * nw;
  int32_t *run = ds + 2;
  int32_t *lm = a.dstate + (int64_t)a.c.batch * (np + 2) + off;
  const int nh = a.c.L * a.H_q;
  int *dist = reinterpret_cast<int *>(sk_s);
  int *run_new = dist + max(p.W, p.p_max);  // the early phase's period runs, committed later

  // ln n and the bounds of the votes (see count_vote and fix_side) for length m: novel rows
  // against theta_ttr w, the stall test's tail against theta_nov stall_len, the entropy sum
  // against theta_ent L H_q ln n, the suffix-mass sum against theta_lift W_s L H_q / n
  auto form_bounds = [&](int m) {
    const double logn = m >= 2 ? log((double)m) : 1.0;
    const int m1 = max(m, 1);
    s_logn = logn;
    s_bound_ttr = count_bounds(p.theta_ttr * (double)min(p.W, m));
    s_bound_stall = count_bounds(p.theta_nov * (double)p.stall_len);
    s_bound_ent = fix_bound(p.theta_ent * (double)nh * logn);
    s_bound_lift = fix_bound(p.theta_lift * (double)min(p.suffix_w, m1) * (double)nh / (double)m1);
  };

  // (0) Before the dependency wait: the comparisons of the new row, which need only the
  // sketches and the monitor state, overlap the end of the kernel before (the attention pass,
  // whose statistics this kernel waits for).  Every read here goes to L2 only (ld.global.cg:
  // nothing is left in L1 for the reads after the wait), stays within the sequence's slots,
  // and writes nothing but shared memory; after the wait the length, the monitor's synced
  // length and the new row are read again, and unless all three are unchanged (the kernel
  // before did not write them) the results are dropped for a recompute.  The one kernel that
  // rewrites window rows without changing any of the three, lg_sketch_build's, lets its
  // successor start only once it has completed.
  // (one read by thread 0, handed on through shared memory: a kernel still writing them could
  // otherwise split the CTA between the two paths)
  if (tid == 0) {
    s_n0 = __ldcg(a.c.len + b);
    s_synced0 = __ldcg(ds);
  }
  __syncthreads();
  const int n0 = s_n0, synced0 = s_synced0;
  const bool pre = n0 >= 1 && synced0 + 1 == n0 && cpr <= kPreRowChunks;
  if (warp == kStatWarps) {
    if (lane == 0) form_bounds(n0);
    if (pre) {
      const uint4 *ri4 = reinterpret_cast<const uint4 *>(sk_g + (int64_t)(n0 - 1) * nw);
      for (int q = lane; q < cpr; q += 32) s_newrow[q] = __ldcg(ri4 + q);
    }
  }
  if (pre) {
    // (2) the new row i against the rows the window and the periods need, [jlo, i), on the
    // warps after the statistics and ln n: chunk q of row j is read by consecutive lanes (rows
    // are contiguous: a warp reads 512 contiguous bytes), all of a thread's loads in flight at
    // once, the chunk popcounts summed per row into dist[] in shared memory (the staging area
    // of the recompute path, unused here); then the latest match, the novel rows and the
    // period runs, reduced per warp and kept in shared memory until they are committed
    const int n = n0, i = n0 - 1;
    const int w = min(p.W, n), wlo = n - w;
    const uint32_t *ri = sk_g + (int64_t)i * nw;
    const int jlo = max(0, min(wlo, i - p.p_max));
    const int m_cnt = i - jlo;
    const int r0 = wlo + tid;
    const int lm0 = r0 < i ? __ldcg(lm + r0) : 0;
    const int run0 = tid < np ? __ldcg(run + tid) : 0;
    const int ct = tid - kCmpWarp0 * 32;  // index among the comparing threads, < 0 elsewhere
    if (ct >= 0) {
      if ((cpr & (cpr - 1)) == 0 && cpr <= 32) {
        // a power-of-two number of chunks: each row's chunks sit in aligned lanes of one warp
        const uint4 *rows4 = reinterpret_cast<const uint4 *>(sk_g + (int64_t)jlo * nw);
        const uint4 *ri4 = reinterpret_cast<const uint4 *>(ri);
        const int total = m_cnt * cpr;
        // a thread's chunk index is ct mod cpr in every row (the stride is a multiple of 32)
        const uint4 v = __ldcg(ri4 + (ct & (cpr - 1)));
        for (int base = 0; base < total; base += kCmpThreads * kCmpBatch) {
          uint4 u[kCmpBatch];
#pragma unroll
          for (int k = 0; k < kCmpBatch; ++k) {
            const int f = base + ct + k * kCmpThreads;
            u[k] = f < total ? __ldcg(rows4 + f) : make_uint4(0u, 0u, 0u, 0u);
          }
#pragma unroll
          for (int k = 0; k < kCmpBatch; ++k) {
            const int f = base + ct + k * kCmpThreads;
            int pc = __popc(u[k].x ^ v.x) + __popc(u[k].y ^ v.y) + __popc(u[k].z ^ v.z) +
                     __popc(u[k].w ^ v.w);
            for (int o = cpr >> 1; o >= 1; o >>= 1) pc += __shfl_xor_sync(0xffffffffu, pc, o);
            if (f < total && (lane & (cpr - 1)) == 0) dist[f / cpr] = pc;
          }
        }
      } else {
        for (int r = ct; r < m_cnt; r += kCmpThreads)
          dist[r] = hamming(ri, sk_g + (int64_t)(jlo + r) * nw, nw);
      }
    }
    __syncthreads();
    int latest = -1;
    for (int j = i - 1 - tid; j >= wlo; j -= kDetectThreads)
      if (dist[j - jlo] <= thr) {
        latest = j;
        break;
      }
    // novel rows of the window other than the new one
    int nov = 0, nov_tail = 0;
    for (int r = r0; r < i; r += kDetectThreads) {
      const int novel = (r == r0 ? lm0 : __ldcg(lm + r)) < wlo;
      nov += novel;
      if (r >= n - p.stall_len) nov_tail += novel;
    }
    // period runs; P ascends with the thread index, so the first qualifying P of a warp is
    // its lowest lane's and a thread's first qualifying P is its smallest
    int pstar = 0x7fffffff;
    for (int pi = tid; pi < np; pi += kDetectThreads) {
      const int P = p.p_min + pi;
      const int cap = max(p.m_rep * P, p.l_min);
      const int j = i - P;
      const bool m = j >= 0 && dist[j - jlo] <= thr;
      const int r = m ? min((pi == tid ? run0 : __ldcg(run + pi)) + 1, cap) : 0;
      run_new[pi] = r;
      if (pstar == 0x7fffffff && n >= cap + P && r >= cap) pstar = P;
    }
    latest = __reduce_max_sync(0xffffffffu, latest);
    nov = __reduce_add_sync(0xffffffffu, nov);
    nov_tail = __reduce_add_sync(0xffffffffu, nov_tail);
    pstar = (int)__reduce_min_sync(0xffffffffu, (unsigned)pstar);
    if (lane == 0) {
      w_latest[warp] = latest;
      w_nov[warp] = nov;
      w_nov_tail[warp] = nov_tail;
      w_pstar[warp] = pstar;
    }
    __syncthreads();
    if (tid == 0) {
      int lt = -1, nv = 0, nt = 0, ps = 0x7fffffff;
      for (int k = 0; k < kDetectWarps; ++k) {
        lt = max(lt, w_latest[k]);
        nv += w_nov[k];
        nt += w_nov_tail[k];
        ps = min(ps, w_pstar[k]);
      }
      s_latest = lt;
      const int novel = lt < wlo;
      s_novel = nv + novel;
      s_novel_tail = nt + (p.stall_len >= 1 ? novel : 0);
      s_pstar = ps;
    }
  }
  pdl_enter();  // the statistics of the kernel before, and every write before it, from here on

  // the sequence's guard state, {t_gen, cd, level, last_trig} and {n_int, pad}, read by the
  // thread that updates it; the device status, decided for the whole CTA at the next barrier
  int4 st_a = make_int4(0, 0, 0, 0), st_b = make_int4(0, 0, 0, 0);
  int bad0 = 0;
  if (tid == 0) {
    bad0 = status_bad(status);
    st_a = reinterpret_cast<const int4 *>(a.state + b)[0];
    st_b = reinterpret_cast<const int4 *>(a.state + b)[1];
  }
  const int B = a.budget[b];

  // (1) sums of the entropies and suffix masses over every layer and head, one warp per SM
  // sub-partition.  The sums are exact in 64-bit fixed point (units of 2^-40: a value loses at
  // most 2^-40 when it is scaled and truncated, and values up to 2^23 fit), on the integer
  // pipes rather than GB300's slow fp64 pipe; a non-finite statistic makes its sum NaN.  The
  // fourth warp reads the length, the synced length and the new row again.
  if (warp < kStatWarps) {
    // kStatBatch loads in flight per thread before the first add (one round trip per batch)
    long long se = 0, sl = 0;
    int finite = 1;
    for (int t0 = tid; t0 < nh; t0 += kStatWarps * 32 * kStatBatch) {
      float4 st[kStatBatch];
#pragma unroll
      for (int k = 0; k < kStatBatch; ++k) {
        const int t = t0 + k * kStatWarps * 32;
        const int layer = t / a.H_q, h = t - layer * a.H_q;
        st[k] = t < nh ? __ldg(reinterpret_cast<const float4 *>(a.stats) +
                               ((int64_t)layer * a.c.batch + b) * a.H_q + h)
                       : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int k = 0; k < kStatBatch; ++k) {
        finite &= isfinite(st[k].z) && isfinite(st[k].w);
        se += __float2ll_rz(st[k].z * kFixScale);
        sl += __float2ll_rz(st[k].w * kFixScale);
      }
    }
    for (int o = 16; o >= 1; o >>= 1) {
      se += __shfl_xor_sync(0xffffffffu, se, o);
      sl += __shfl_xor_sync(0xffffffffu, sl, o);
    }
    finite = __all_sync(0xffffffffu, finite);
    if (lane == 0) {
      red_e[warp] = se;
      red_l[warp] = sl;
      red_ok[warp] = finite;
    }
  } else if (warp == kStatWarps) {
    int ok = 1;
    if (lane == 0) {
      const int n1 = __ldcg(a.c.len + b);
      s_n = n1;
      ok = n1 == n0 && __ldcg(ds) == synced0;
    }
    if (pre) {
      const uint4 *ri4 = reinterpret_cast<const uint4 *>(sk_g + (int64_t)(n0 - 1) * nw);
      for (int q = lane; q < cpr; q += 32) {
        const uint4 x = __ldcg(ri4 + q), y = s_newrow[q];
        ok &= x.x == y.x && x.y == y.y && x.z == y.z && x.w == y.w;
      }
    }
    ok = __all_sync(0xffffffffu, ok);
    if (lane == 0) s_valid = pre && ok;
  }
  if (tid == 0) s_bad = bad0;
  __syncthreads();
  if (s_bad) return;  // the same decision in every thread of the CTA
  const int n = s_n;
  const int w = min(p.W, n);
  const int wlo = n - w;

  if (s_valid) {
    // the early phase stands: commit its period runs and the new row's latest match
    for (int pi = tid; pi < np; pi += kDetectThreads) run[pi] = run_new[pi];
    if (tid == 0) lm[n - 1] = s_latest;
  } else {
    // (2') recompute (first call, after a prune or any other change of the cache, or when the
    // early phase's inputs changed): every window row's latest match, every period's trailing
    // run, from rows staged in shared memory
    const int lo_s = max(0, n - a.smem_rows);
    for (int t = tid; t < (n - lo_s) * nw; t += kDetectThreads) {
      const int r = t / nw;
      sk_s[r * stride + (t - r * nw)] = sk_g[(int64_t)lo_s * nw + t];
    }
    if (tid == 0) {
      s_novel = 0;
      s_novel_tail = 0;
      s_pstar = 0x7fffffff;
      if (n != n0) form_bounds(n);
    }
    __syncthreads();
    auto row = [=](int r) -> const uint32_t * {
      return r >= lo_s ? sk_s + (int64_t)(r - lo_s) * stride : sk_g + (int64_t)r * nw;
    };
    for (int r = wlo + warp; r < n; r += kDetectWarps) {
      // latest j in [wlo, r) whose row matches row r, or -1 (one warp, nearest rows first)
      const uint32_t *rr = row(r);
      int found = -1;
      for (int top = r - 1; top >= wlo; top -= 32) {
        const int j = top - lane;
        const bool m = j >= wlo && rows_match(rr, row(j), nw, thr);
        const unsigned bal = __ballot_sync(0xffffffffu, m);
        if (bal) {
          found = top - (__ffs(bal) - 1);
          break;
        }
      }
      if (lane == 0) lm[r] = found;
    }
    for (int pi = warp; pi < np; pi += kDetectWarps) {
      const int P = p.p_min + pi;
      const int cap = max(p.m_rep * P, p.l_min);
      int r = cap;
      for (int k0 = 0; k0 < cap; k0 += 32) {
        const int k = k0 + lane;
        const int i = n - 1 - k;
        const bool ok = k < cap && i - P >= 0 && rows_match(row(i), row(i - P), nw, thr);
        const unsigned bad = __ballot_sync(0xffffffffu, !ok);
        if (bad) {
          r = min(cap, k0 + __ffs(bad) - 1);
          break;
        }
      }
      if (lane == 0) run[pi] = r;
    }
    __syncthreads();
    int nov = 0, nov_tail = 0;
    for (int r = wlo + tid; r < n; r += kDetectThreads) {
      const int novel = lm[r] < wlo;
      nov += novel;
      if (r >= n - p.stall_len) nov_tail += novel;
    }
    nov = __reduce_add_sync(0xffffffffu, nov);
    nov_tail = __reduce_add_sync(0xffffffffu, nov_tail);
    if (lane == 0 && nov) atomicAdd(&s_novel, nov);
    if (lane == 0 && nov_tail) atomicAdd(&s_novel_tail, nov_tail);
    for (int pi = tid; pi < np; pi += kDetectThreads) {
      const int P = p.p_min + pi;
      const int span_len = max(p.m_rep * P, p.l_min);
      if (n >= span_len + P && run[pi] >= span_len) atomicMin(&s_pstar, P);
    }
    __syncthreads();
  }
  // (3) the votes, the stall gate and the trigger, on thread 0, against the bounds formed in (0)
  // (again after the wait when the length changed; count_vote, fix_side), then the guard state's
  // update.  The recompute path's counts arrive by shared-memory atomics (its own barrier above);
  // the early phase's are thread 0's own.
  if (tid == 0) {
    int trig = 0, sig1 = 0, sig2 = 0, sig3 = 0, stall = 0;
    const bool tailrep = s_pstar != 0x7fffffff;
    long long e_fix = 0, l_fix = 0;
    int ok = 1;
    if (n >= 1) {
      for (int k = 0; k < kStatWarps; ++k) {
        e_fix += red_e[k];
        l_fix += red_l[k];
        ok &= red_ok[k];
      }
      sig1 = count_vote(s_novel, s_bound_ttr, w, p.theta_ttr);
      stall = w >= p.stall_len && p.stall_len > 0 &&
              count_vote(s_novel_tail, s_bound_stall, p.stall_len, p.theta_nov);
      if (n < 2) {
        sig2 = 1.0 < p.theta_ent;  // the mean is taken as 1 below two rows
      } else if (ok) {
        const int side = fix_side(e_fix, s_bound_ent);
        sig2 = side ? side < 0 : sum_quotient_vote(e_fix, 1, (double)nh, s_logn, p.theta_ent, 0);
      }
      if (ok) {
        const int side = fix_side(l_fix, s_bound_lift);
        sig3 = side ? side > 0
                    : sum_quotient_vote(l_fix, n, (double)min(p.suffix_w, n), (double)nh,
                                        p.theta_lift, 1);
      }
      trig = st_a.x >= p.t_min && st_a.y == 0 && sig1 + sig2 + sig3 >= p.K && (stall || tailrep);
    }
    if (a.diag && n >= 1) {
      // the quotients themselves (tests and diagnostics only): mean H / ln n, mean S n / W_s,
      // novel-row fraction
      double *dg = a.diag + 8 * b;
      const double e_sum = ok ? (double)e_fix * kFixUnit : (double)NAN;
      const double l_sum = ok ? (double)l_fix * kFixUnit : (double)NAN;
      dg[0] = n >= 2 ? e_sum / ((double)nh * s_logn) : 1.0;
      dg[1] = l_sum * (double)n / ((double)min(p.suffix_w, n) * (double)nh);
      dg[2] = (double)s_novel / (double)w;
      dg[3] = sig1;
      dg[4] = sig2;
      dg[5] = sig3;
      dg[6] = stall;
      dg[7] = tailrep ? s_pstar : 0;
    }
    // state: x = t_gen, y = cd, z = level, w = last_trig; st_b.x = n_int
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
    ds[0] = n;
    a.flags[b] = trig;
    if (!(trig && tailrep)) {
      a.spans[2 * b] = 0;
      a.spans[2 * b + 1] = 0;
      s_span_lo = 0;
      s_span_hi = 0;
    }
    s_level = st_a.z;
    s_trig = trig;
    s_mismatch = -1;
  }
  __syncthreads();

  // (4) span: extend the verified tail back while rows keep matching the row P* earlier
  const int trig = s_trig;
  const int Pstar = s_pstar;
  const int R = B / 2;
  if (trig && Pstar != 0x7fffffff) {
    const int span_len = max(p.m_rep * Pstar, p.l_min);
    const int lo_ext = max(Pstar, n - R);
    int s = n - span_len;
    if (s < lo_ext) {
      s = lo_ext;
    } else {
      for (int hi = s; hi > lo_ext; hi -= kDetectThreads) {
        const int i = hi - 1 - tid;
        if (i >= lo_ext && hamming(sk_g + (int64_t)i * nw, sk_g + (int64_t)(i - Pstar) * nw, nw) > thr)
          atomicMax(&s_mismatch, i);
        __syncthreads();
        const int found = s_mismatch;
        __syncthreads();
        if (found >= 0) break;
      }
      if (s_mismatch >= 0) s = s_mismatch + 1;
      else s = lo_ext;
    }
    if (tid == 0) {
      const int lo = max(max(s - Pstar, n - R), 0);
      a.spans[2 * b] = lo;
      a.spans[2 * b + 1] = n;
      s_span_lo = lo;
      s_span_hi = n;
    }
  }
  if (a.kept_idx) {
    // (5) the retained set of this sequence from the decision just taken; a sequence that
    // neither triggered nor outgrew its budget only marks "no prune"
    int code = 0;
    if (trig || n > B) {
      __syncthreads();  // thread 0's span and level
      code = write_keep(a.c, b, n, B, trig, s_span_lo, s_span_hi, s_level, p, a.kept_idx,
                        a.kept_count, a.max_keep, a.max_len, tid, kDetectThreads);
    } else if (tid == 0) {
      a.kept_count[b] = -1;
    }
    if (code && tid == 0) set_status(a.c.dev_status, code);
  }
}

int detect_smem_rows(const lg_guard_params &p) {
  const int tail = max(p.m_rep * p.p_max, p.l_min) + p.p_max;
  return max(p.W, tail);
}

size_t detect_smem_bytes(const lg_guard_params &p, int nwords) {
  return (size_t)detect_smem_rows(p) * (nwords + 1) * 4;
}

size_t detect_state_bytes(const lg_cache &c, const lg_guard_params &p) {
  const int64_t np = p.p_max - p.p_min + 1;
  return (size_t)((int64_t)c.batch * (np + 2) + c.S_total) * sizeof(int32_t);
}

// ------------------------------------------------------------------ retained set I_keep

struct KeepArgs {
  lg_cache c;
  const int32_t *flags, *spans;
  const lg_guard_state *state;
  const int32_t *budget;
  lg_guard_params p;
  int32_t *kept_idx, *kept_count;
  int max_keep, max_len;
};

constexpr int kKeepThreads = 1024;

__global__ void __launch_bounds__(kKeepThreads) keep_set_kernel(KeepArgs a) {
  pdl_enter();
  const int b = blockIdx.x, tid = threadIdx.x;
  const int32_t *status = a.c.dev_status;
  const int n = a.c.len[b];
  const int B = a.budget[b];
  const int flag = a.flags ? a.flags[b] : 0;
  const int span_lo = a.spans ? a.spans[2 * b] : 0, span_hi = a.spans ? a.spans[2 * b + 1] : 0;
  const int level = a.flags ? a.state[b].level : 0;  // state may be null without flags
  if (status_bad(status)) return;
  const int code = write_keep(a.c, b, n, B, flag, span_lo, span_hi, level, a.p, a.kept_idx,
                              a.kept_count, a.max_keep, a.max_len, tid, kKeepThreads);
  if (code && tid == 0) set_status(a.c.dev_status, code);
}

// ------------------------------------------------------------------ ordered in-place gather

constexpr int kCompactThreads = 256;
constexpr int kCompactStageBytes = 16384;  // one tile of destination rows
constexpr int kCompactStages = 4;          // ring of tiles: three gathers in flight, one store
constexpr int kCompactChunks = kCompactStageBytes / 16 / kCompactThreads;  // 16-byte chunks
constexpr int kCompactSeqList = 1024;  // pruned sequences listed in shared memory up to this batch
constexpr size_t kCompactSmem = (size_t)kCompactStages * kCompactStageBytes;

// Stream (sequence b, one of 2*L*H_kv K/V streams or the sketch stream): slot j <- row kept[j]
// for j >= j0, in tiles of kCompactStageBytes of destination rows, ascending.  CTAs take
// (sequence, stream) items of the pruned sequences grid-stride (each CTA first lists them from
// one pass over kept_count, so a step that prunes nothing costs that pass).
//
// A tile is gathered row chunk by row chunk with 16-byte asynchronous copies into a ring of
// shared-memory stages (kCompactStages - 1 tiles in flight, no registers held), then written
// back by one bulk copy of the whole tile's contiguous slots.  In place and race-free without
// any further ordering: kept[] is strictly increasing with kept[j] >= j, so a row read for tile
// i' > i lies at or above kept[first slot of i'] > every slot of tile i, and every row a slot of
// tile i is read for (kept[j] = s means j <= s) belongs to a tile <= i, whose copies have all
// landed in shared memory before tile i's store is issued (the wait and the barrier below).
__global__ void __launch_bounds__(kCompactThreads) compact_kernel(lg_cache c,
                                                                  const int32_t *kept_idx,
                                                                  const int32_t *kept_count,
                                                                  int max_keep) {
  pdl_enter();
  extern __shared__ __align__(128) unsigned char s_stage[];  // kCompactStages tiles
  __shared__ int s_seq[kCompactSeqList], s_cnt[kCompactSeqList];
  __shared__ int s_wtot[kCompactThreads / 32];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int row_bytes_kv = c.d * (c.dtype == LG_BF16 ? 2 : 4);
  const int nwords = c.H_kv * c.d / 32;
  const int n_kv = 2 * c.L * c.H_kv;
  const int per_seq = n_kv + 1;
  // the pruned sequences and their counts, in sequence order (read before the status word)
  const bool listed = c.batch <= kCompactSeqList;
  int n_listed = 0;
  __shared__ int s_bad;
  // the device status, read beside the kept counts and decided after the listing's barrier
  const int bad0 = tid == 0 ? (int)status_bad(c.dev_status) : 0;
  if (listed) {
    for (int b0 = 0; b0 < c.batch; b0 += kCompactThreads) {
      const int b = b0 + tid;
      const int k = b < c.batch ? kept_count[b] : -1;
      const unsigned bal = __ballot_sync(0xffffffffu, k >= 0);
      if (lane == 0) s_wtot[warp] = __popc(bal);
      __syncthreads();
      int at = n_listed, tot = 0;
      for (int w = 0; w < kCompactThreads / 32; ++w) {
        at += w < warp ? s_wtot[w] : 0;
        tot += s_wtot[w];
      }
      if (k >= 0) {
        at += __popc(bal & ((1u << lane) - 1u));
        s_seq[at] = b;
        s_cnt[at] = k;
      }
      n_listed += tot;
      if (b0 + kCompactThreads >= c.batch && tid == 0) s_bad = bad0;
      __syncthreads();
    }
  } else {
    if (tid == 0) s_bad = bad0;
    __syncthreads();
  }
  if (s_bad) return;  // the same decision in every thread of the CTA
  const int n_items = (listed ? n_listed : c.batch) * per_seq;
  // grid-stride over (sequence, stream)
  for (int item = blockIdx.x; item < n_items; item += gridDim.x) {
    const int r = item / per_seq, stream = item - r * per_seq;
    const int b = listed ? s_seq[r] : r;
    const int cnt = listed ? s_cnt[r] : kept_count[b];
    if (cnt < 0) continue;
    unsigned char *base;
    int row_bytes;
    if (stream < n_kv) {
      const int lh = stream >> 1;
      unsigned char *t = (unsigned char *)((stream & 1) ? c.v : c.k);
      base = t + ((int64_t)lh * c.S_total + c.seq_off[b]) * row_bytes_kv;
      row_bytes = row_bytes_kv;
    } else {
      if (!c.sketch) continue;
      base = (unsigned char *)(c.sketch + c.seq_off[b] * nwords);
      row_bytes = nwords * 4;
    }
    const int32_t *kept = kept_idx + (int64_t)b * max_keep;
    // first slot that moves: kept[j] == j exactly for j < j0 (and kept[j] > j after), found by
    // a 32-way search in every warp (the same result in all)
    int lo = 0, hi = cnt;
    while (lo < hi) {
      const int step = (hi - lo + 31) >> 5;
      const int x = lo + lane * step;
      const unsigned m = __ballot_sync(0xffffffffu, x < hi && kept[x] != x);
      if (m) {
        const int f = __ffs(m) - 1;
        hi = lo + f * step;
        if (f) lo += (f - 1) * step + 1;
      } else {
        lo += min(31, (hi - 1 - lo) / step) * step + 1;
      }
    }
    const int j0 = lo;
    const int cpr = row_bytes >> 4;
    const int T = kCompactStageBytes / row_bytes;  // rows per tile
    const int n_tiles = (cnt - j0 + T - 1) / T;
    if (n_tiles <= 0) continue;
    // this thread's chunks of a tile: row within the tile and byte offset within the row; in
    // the stage a chunk sits at its chunk index x 16 (the tile's rows back to back)
    int c_row[kCompactChunks], c_off[kCompactChunks], kv[kCompactChunks];
#pragma unroll
    for (int k = 0; k < kCompactChunks; ++k) {
      const int ci = k * kCompactThreads + tid;
      c_row[k] = ci / cpr;
      c_off[k] = (ci - c_row[k] * cpr) * 16;
    }
    // kv[k] <- source row of chunk k of tile p (requested a tile ahead of its copies)
    auto fetch_rows = [&](int p) {
      const int t0 = j0 + p * T, rows = min(T, cnt - t0);
#pragma unroll
      for (int k = 0; k < kCompactChunks; ++k)
        kv[k] = (p < n_tiles && c_row[k] < rows) ? kept[t0 + c_row[k]] : 0;
    };
    auto gather = [&](int p) {
      const int t0 = j0 + p * T, rows = min(T, cnt - t0);
      unsigned char *st = s_stage + (p % kCompactStages) * kCompactStageBytes;
#pragma unroll
      for (int k = 0; k < kCompactChunks; ++k)
        if (c_row[k] < rows)
          cp_async16(st + (k * kCompactThreads + tid) * 16,
                     base + (int64_t)kv[k] * row_bytes + c_off[k]);
    };
    for (int p = 0; p < kCompactStages - 1; ++p) {
      if (p < n_tiles) {
        fetch_rows(p);
        gather(p);
      }
      cp_async_commit();  // one group per tile, empty past the end (uniform group counting)
    }
    fetch_rows(kCompactStages - 1);
    for (int i = 0; i < n_tiles; ++i) {
      cp_async_wait<kCompactStages - 2>();  // this thread's copies of tile i have landed
      fence_proxy_async_smem();
      if (tid == 0) bulk_wait_read_all();  // tile i-1's store has read its stage
      __syncthreads();
      if (tid == 0) {
        const int t0 = j0 + i * T, rows = min(T, cnt - t0);
        bulk_store(base + (int64_t)t0 * row_bytes,
                   s_stage + (i % kCompactStages) * kCompactStageBytes,
                   (uint32_t)(rows * row_bytes));
        bulk_commit();
      }
      const int p = i + kCompactStages - 1;  // into the stage tile i-1 used
      if (p < n_tiles) gather(p);
      cp_async_commit();
      fetch_rows(p + 1);
    }
    // the next item's first copies reuse the stages
    if (tid == 0) bulk_wait_read_all();
    __syncthreads();
  }
  if (tid == 0) bulk_wait_all();
}

// ------------------------------------------------------------------ H2O comparator

__global__ void h2o_reset_kernel(lg_cache c, int max_len) {
  pdl_enter();
  const int lh = blockIdx.y, b = blockIdx.z;
  const int n = min(c.len[b], max_len);
  const int64_t o = (int64_t)lh * c.S_total + c.seq_off[b];
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) {
    c.pos[o + i] = i;
    c.h2o[o + i] = 0.f;
  }
}

__device__ __forceinline__ uint64_t h2o_key(float score, int32_t pos) {
  uint32_t u = __float_as_uint(score);
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);  // order-preserving
  return ((uint64_t)u << 32) | (uint32_t)pos;
}

constexpr int kH2OThreads = 256;
constexpr int kH2OTile = 32;
constexpr int kH2OMaxQ = 2 * kH2OTile * 32 / kH2OThreads;  // 16-byte chunks per thread, 512 B rows

// One CTA per (sequence, layer, kv-head) stream of a sequence over budget.
// kMode kEvictH2O: keep the recent half of the budget and the highest (score, pos) rows.
// kMode kEvictStreaming: keep positions < n_sink and the budget - n_sink most recent ones.
enum { kEvictH2O = 0, kEvictStreaming = 1 };

template <int kMode>
__global__ void __launch_bounds__(kH2OThreads) evict_kernel(lg_cache c, const int32_t *budget,
                                                            const int32_t *pos_now, int max_len,
                                                            int n_sink) {
  pdl_enter();
  __shared__ unsigned long long s_wbest[kH2OThreads / 32];
  __shared__ int s_wslot[kH2OThreads / 32];
  __shared__ int s_slot, s_count, s_out;
  __shared__ unsigned int hist[256];
  __shared__ unsigned long long s_prefix;
  __shared__ int s_remaining;
  const int lh = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  if (cta_status_bad(c.dev_status)) return;
  const int n = c.len[b], B = budget[b];
  if (n <= B) return;
  if (n > max_len) {
    if (tid == 0) set_status(c.dev_status, LG_ERR_CAPACITY);
    return;
  }
  // recent: pos > thrp (H2O: the newest B/2 positions; streaming: the newest B - n_sink)
  const int32_t thrp = pos_now[b] - (kMode == kEvictH2O ? B / 2 : B - n_sink);
  const int64_t o = (int64_t)lh * c.S_total + c.seq_off[b];
  float *sc = c.h2o + o;
  int32_t *ps = c.pos + o;
  const int rb = c.d * (c.dtype == LG_BF16 ? 2 : 4);
  const int cpr = rb / 16;
  uint4 *K4 = reinterpret_cast<uint4 *>((unsigned char *)c.k + o * rb);
  uint4 *V4 = reinterpret_cast<uint4 *>((unsigned char *)c.v + o * rb);

  // eviction order among the rows outside the protected set: lowest key first
  auto evict_key = [&](int i) -> unsigned long long {
    return kMode == kEvictH2O ? (unsigned long long)h2o_key(sc[i], ps[i])
                              : (unsigned long long)(uint32_t)ps[i];
  };
  auto protected_row = [&](int i) -> bool {
    return ps[i] > thrp || (kMode == kEvictStreaming && ps[i] < n_sink);
  };
  auto refill = [&](int x) {  // slot x takes the last slot's row, score and position
    for (int ch = tid; ch < cpr; ch += kH2OThreads) {
      K4[(int64_t)x * cpr + ch] = K4[(int64_t)(n - 1) * cpr + ch];
      V4[(int64_t)x * cpr + ch] = V4[(int64_t)(n - 1) * cpr + ch];
    }
    if (tid == 0) {
      sc[x] = sc[n - 1];
      ps[x] = ps[n - 1];
    }
  };
  if (kMode == kEvictStreaming && n == B + 1 && B > n_sink) {
    // Sliding window: after the first cut its slots [n_sink, B) hold consecutive positions in
    // slot order, and each step's row takes the slot of the oldest, so the slots stay a ring in
    // position order and the row to evict (position thrp) sits at n_sink + (thrp - ps[n_sink])
    // mod (B - n_sink).  One check of that slot's position replaces the scan below, which
    // runs whenever the check fails (the same slot in every case the ring holds).
    const int w = B - n_sink;
    const int64_t r = ((int64_t)thrp - ps[n_sink]) % w;
    const int x = n_sink + (int)(r < 0 ? r + w : r);
    if (ps[x] == thrp) {
      refill(x);
      return;
    }
  }
  if (n == B + 1) {
    // one row over budget: evict the lowest key outside the protected rows and refill its
    // slot from the last slot.  Keys are unique (the position is part of the key), so one pass
    // keeps each thread's lowest key with its slot, and a reduction picks the CTA's.
    unsigned long long best = ~0ull;
    int slot = -1;
    for (int i = tid; i < n; i += kH2OThreads)
      if (!protected_row(i)) {
        const unsigned long long key = evict_key(i);
        if (key < best) {
          best = key;
          slot = i;
        }
      }
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
      const unsigned long long ob = __shfl_xor_sync(0xffffffffu, best, o);
      const int os = __shfl_xor_sync(0xffffffffu, slot, o);
      if (ob < best) {
        best = ob;
        slot = os;
      }
    }
    if ((tid & 31) == 0) {
      s_wbest[tid >> 5] = best;
      s_wslot[tid >> 5] = slot;
    }
    __syncthreads();
    if (tid == 0) {
      unsigned long long m = ~0ull;
      int x = -1;
      for (int w = 0; w < kH2OThreads / 32; ++w)
        if (s_wbest[w] < m) {
          m = s_wbest[w];
          x = s_wslot[w];
        }
      s_slot = x;
    }
    __syncthreads();
    const int x = s_slot;
    if (x < 0 || x == n - 1) return;
    refill(x);
    return;
  }
  if (kMode == kEvictStreaming) {
    // closed form: sinks and the newest B - n_sink positions
    if (tid == 0) s_out = 0;
    __syncthreads();
  }

  // cut to B rows: recent rows plus the k = B - n_recent highest keys among the others
  int k = 0;
  unsigned long long kth = 0;
  if (kMode == kEvictH2O) {
  if (tid == 0) s_count = 0;
  __syncthreads();
  int cnt_local = 0;
  for (int i = tid; i < n; i += kH2OThreads) cnt_local += ps[i] > thrp;
  atomicAdd(&s_count, cnt_local);
  if (tid == 0) {
    s_prefix = 0;
    s_out = 0;
  }
  __syncthreads();
  k = B - s_count;
  unsigned long long mask = 0;
  if (tid == 0) s_remaining = k;
  for (int digit = 7; digit >= 0; --digit) {
    hist[tid] = 0;
    __syncthreads();
    const unsigned long long prefix = s_prefix;
    for (int i = tid; i < n; i += kH2OThreads) {
      if (ps[i] > thrp) continue;
      const unsigned long long key = h2o_key(sc[i], ps[i]);
      if ((key & mask) == prefix) atomicAdd(&hist[(key >> (8 * digit)) & 255u], 1u);
    }
    __syncthreads();
    if (tid == 0) {
      int rem = s_remaining, cum = 0, v = 255;
      for (; v > 0; --v) {
        if (cum + (int)hist[v] >= rem) break;
        cum += hist[v];
      }
      s_remaining = rem - cum;
      s_prefix = prefix | ((unsigned long long)v << (8 * digit));
    }
    mask |= 255ull << (8 * digit);
    __syncthreads();
  }
  kth = s_prefix;  // key of the k-th highest non-recent row
  }

  // ordered compaction of K, V, score and pos over source tiles of kH2OTile rows
  const int lane = tid & 31, warp = tid >> 5;
  for (int t0 = 0; t0 < n; t0 += kH2OTile) {
    __shared__ int s_dest[kH2OTile];
    __shared__ int s_tile_kept;
    if (warp == 0) {
      const int i = t0 + lane;
      bool keep = false;
      if (i < n)
        keep = protected_row(i) || (kMode == kEvictH2O && k > 0 && h2o_key(sc[i], ps[i]) >= kth);
      const unsigned bal = __ballot_sync(0xffffffffu, keep);
      s_dest[lane] = keep ? s_out + __popc(bal & ((1u << lane) - 1u)) : -1;
      if (lane == 0) s_tile_kept = __popc(bal);
    }
    __syncthreads();
    // each thread moves chunks of the kept rows of this tile
    uint4 kv[kH2OMaxQ];
    float scv = 0.f;
    int32_t psv = 0;
    const int nchunks = kH2OTile * cpr;  // per tensor
#pragma unroll
    for (int q = 0; q < kH2OMaxQ; ++q) {
      const int ci = q * kH2OThreads + tid;
      const int tensor = ci / nchunks, rc = ci % nchunks;
      const int r = rc / cpr, ch = rc % cpr;
      if (tensor < 2 && s_dest[r] >= 0 && t0 + r != s_dest[r]) {
        const uint4 *src = tensor ? V4 : K4;
        kv[q] = src[(int64_t)(t0 + r) * cpr + ch];
      }
    }
    if (tid < kH2OTile && s_dest[tid] >= 0) {
      scv = sc[t0 + tid];
      psv = ps[t0 + tid];
    }
    __syncthreads();
#pragma unroll
    for (int q = 0; q < kH2OMaxQ; ++q) {
      const int ci = q * kH2OThreads + tid;
      const int tensor = ci / nchunks, rc = ci % nchunks;
      const int r = rc / cpr, ch = rc % cpr;
      if (tensor < 2 && s_dest[r] >= 0 && t0 + r != s_dest[r]) {
        uint4 *dst = tensor ? V4 : K4;
        dst[(int64_t)s_dest[r] * cpr + ch] = kv[q];
      }
    }
    if (tid < kH2OTile && s_dest[tid] >= 0) {
      sc[s_dest[tid]] = scv;
      ps[s_dest[tid]] = psv;
    }
    if (tid == 0) s_out += s_tile_kept;
    __syncthreads();
  }
}

__global__ void h2o_len_kernel(lg_cache c, const int32_t *budget) {
  pdl_enter();
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= c.batch || status_bad(c.dev_status)) return;
  if (c.len[b] > budget[b]) c.len[b] = budget[b];
}

// ------------------------------------------------------------------ launchers

cudaError_t launch_begin_step(const lg_cache &c, cudaStream_t s) {
  LG_TRY(launch_pdl(begin_step_kernel, (c.batch + 127) / 128, 128, 0, s, c));
  return cudaGetLastError();
}

cudaError_t launch_append(const lg_cache &c, int layer0, int n_layers, const void *k_new,
                          const void *v_new, const int32_t *pos_new, int guard_layer,
                          cudaStream_t s) {
  const int cpr = c.d * (c.dtype == LG_BF16 ? 2 : 4) / 16;
  const int64_t total = (int64_t)n_layers * c.batch * c.H_kv * cpr;
  const int row_blocks = (int)((total + 255) / 256);
  const bool sk = c.sketch && guard_layer >= layer0 && guard_layer < layer0 + n_layers;
  const int grid = row_blocks + (sk ? c.batch : 0);
  if (c.dtype == LG_BF16) {
    LG_TRY(launch_pdl(append_kernel<__nv_bfloat16>, grid, 256, 0, s, c, layer0, n_layers,
                      (const uint4 *)k_new, (const uint4 *)v_new, pos_new, row_blocks,
                      guard_layer - layer0));
  } else {
    LG_TRY(launch_pdl(append_kernel<float>, grid, 256, 0, s, c, layer0, n_layers,
                      (const uint4 *)k_new, (const uint4 *)v_new, pos_new, row_blocks,
                      guard_layer - layer0));
  }
  return cudaGetLastError();
}

cudaError_t launch_sketch_build(const lg_cache &c, int guard_layer, int max_len, cudaStream_t s) {
  const int nwords = c.H_kv * c.d / 32;
  int64_t per_seq = (int64_t)max_len * nwords;
  int gx = (int)((per_seq + 255) / 256);
  if (gx > 1024) gx = 1024;
  if (gx < 1) gx = 1;
  dim3 grid(gx, c.batch);
  if (c.dtype == LG_BF16) {
    LG_TRY(launch_pdl(sketch_build_kernel<__nv_bfloat16>, grid, 256, 0, s, c, guard_layer,
                      max_len));
  } else {
    LG_TRY(launch_pdl(sketch_build_kernel<float>, grid, 256, 0, s, c, guard_layer, max_len));
  }
  return cudaGetLastError();
}

cudaError_t launch_state_init(const lg_cache &c, lg_guard_state *state, int t_gen0, cudaStream_t s) {
  LG_TRY(launch_pdl(state_init_kernel, (c.batch + 127) / 128, 128, 0, s, c.batch, state, t_gen0));
  return cudaGetLastError();
}

cudaError_t launch_detect(const lg_cache &c, const float *stats, int H_q, lg_guard_state *state,
                          const int32_t *budget, const lg_guard_params &p, int32_t *flags,
                          int32_t *spans, double *diag, void *dstate, int32_t *kept_idx,
                          int32_t *kept_count, int max_keep, int max_len, cudaStream_t s) {
  DetectArgs a;
  a.kept_idx = kept_idx;
  a.kept_count = kept_count;
  a.max_keep = max_keep;
  a.max_len = max_len;
  a.c = c;
  a.stats = stats;
  a.H_q = H_q;
  a.state = state;
  a.budget = budget;
  a.p = p;
  a.flags = flags;
  a.spans = spans;
  a.diag = diag;
  a.dstate = (int32_t *)dstate;
  a.nwords = c.H_kv * c.d / 32;
  a.thr = (int)floor(p.tau_ham * (double)(a.nwords * 32));
  a.smem_rows = detect_smem_rows(p);
  const size_t smem = detect_smem_bytes(p, a.nwords);
  cudaError_t e = cudaFuncSetAttribute(detect_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)smem);
  if (e != cudaSuccess) return e;
  LG_TRY(launch_pdl(detect_kernel, c.batch, kDetectThreads, smem, s, a));
  return cudaGetLastError();
}

cudaError_t launch_prune_compact(const lg_cache &c, const int32_t *flags, const int32_t *spans,
                                 const lg_guard_state *state, const int32_t *budget,
                                 const lg_guard_params &p, int32_t *kept_idx,
                                 int32_t *kept_count, int max_keep, int max_len, cudaStream_t s) {
  KeepArgs a;
  a.c = c;
  a.flags = flags;
  a.spans = spans;
  a.state = state;
  a.budget = budget;
  a.p = p;
  a.kept_idx = kept_idx;
  a.kept_count = kept_count;
  a.max_keep = max_keep;
  a.max_len = max_len;
  LG_TRY(launch_pdl(keep_set_kernel, c.batch, kKeepThreads, 0, s, a));
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return launch_compact(c, kept_idx, kept_count, max_keep, s);
}

cudaError_t launch_compact(const lg_cache &c, const int32_t *kept_idx, const int32_t *kept_count,
                           int max_keep, cudaStream_t s) {
  // one wave of resident CTAs (items are handed out grid-stride, so a second wave would start
  // its items late); the residency per SM is looked up once per device
  constexpr int kMaxDev = 64;
  static std::atomic<int> resident[kMaxDev];  // CTAs per GPU, 0 = not looked up yet
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) dev = 0;
  int ctas = dev < kMaxDev ? resident[dev].load(std::memory_order_relaxed) : 0;
  if (ctas <= 0) {
    int sms = 152, per_sm = 1;
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    LG_TRY(cudaFuncSetAttribute(compact_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)kCompactSmem));
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, compact_kernel, kCompactThreads,
                                                      kCompactSmem) != cudaSuccess || per_sm < 1)
      per_sm = 1;
    ctas = sms * per_sm;
    if (dev < kMaxDev) resident[dev].store(ctas, std::memory_order_relaxed);
  }
  const int items = c.batch * (2 * c.L * c.H_kv + 1);
  const int grid = items < ctas ? items : ctas;
  LG_TRY(launch_pdl(compact_kernel, grid, kCompactThreads, kCompactSmem, s, c, kept_idx,
                    kept_count, max_keep));
  return cudaGetLastError();
}

cudaError_t launch_h2o_reset(const lg_cache &c, int max_len, cudaStream_t s) {
  int gx = (max_len + 255) / 256;
  if (gx > 256) gx = 256;
  if (gx < 1) gx = 1;
  LG_TRY(launch_pdl(h2o_reset_kernel, dim3(gx, c.L * c.H_kv, c.batch), 256, 0, s, c, max_len));
  return cudaGetLastError();
}

cudaError_t launch_h2o_evict(const lg_cache &c, const int32_t *budget, const int32_t *pos_now,
                             int max_len, cudaStream_t s) {
  LG_TRY(launch_pdl(evict_kernel<kEvictH2O>, dim3(c.L * c.H_kv, c.batch), kH2OThreads, 0, s, c,
                    budget, pos_now, max_len, 0));
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  LG_TRY(launch_pdl(h2o_len_kernel, (c.batch + 127) / 128, 128, 0, s, c, budget));
  return cudaGetLastError();
}

}  // namespace lg

namespace lg {

cudaError_t launch_streaming_evict(const lg_cache &c, const int32_t *budget,
                                   const int32_t *pos_now, int n_sink, int max_len,
                                   cudaStream_t s) {
  LG_TRY(launch_pdl(evict_kernel<kEvictStreaming>, dim3(c.L * c.H_kv, c.batch), kH2OThreads, 0, s,
                    c, budget, pos_now, max_len, n_sink));
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  LG_TRY(launch_pdl(h2o_len_kernel, (c.batch + 127) / 128, 128, 0, s, c, budget));
  return cudaGetLastError();
}

}  // namespace lg
