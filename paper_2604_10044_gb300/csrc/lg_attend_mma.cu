// Decode attention over a bf16 KV cache fused with the guard's per-head statistics (LoopGuard
// Sec. 3.1, Eq. 1; statistics read by Sec. 5.2), on tensor cores.
//
// Persistent CTAs (one per SM) start on chunks blockIdx.x and blockIdx.x + gridDim.x and take
// further chunks from a shared counter, each a run of consecutive rows of one (layer,
// sequence, kv-head), sized in the kernel from the lengths of the call (3 to 16 chunks per
// CTA).  A producer warp streams 128-row K and V tiles into a 3-stage shared-memory ring with
// 2-D tensor copies (cp.async.bulk.tensor, 128-byte swizzle, one box per 64 columns)
// completing on mbarriers.  Each of four consumer warps owns 32 rows of a tile and all g query
// heads of the kv-head (padded to 8):
//   S^T[16 rows x 8 heads] = K[16 x d] q^T      mma.sync m16n8k16 bf16 -> fp32, A by ldmatrix
//   online softmax in log2 units on the accumulator fragments (exact running max per head)
//   o^T[d x 8 heads] += V^T[d x 16 rows] P^T    A by ldmatrix.trans, B = P^T by movmatrix,
//                                               P split into bf16 hi + lo (two MMAs)
// The suffix mass, the entropy term and the normaliser accumulate beside the softmax.  At the
// end of a chunk each warp leaves its own {M, l, u, sigma, o[d]} per head in a shared-memory
// ticket buffer and goes on streaming (no barrier among the consumers); one of four merger
// warps merges the four into the chunk's partial, counts the arrivals of its (layer,
// sequence, kv-head) group, and the arrival that completes a group merges the group's chunk
// partials into out and the statistics.  Rows past the end of a sequence (ragged last tile)
// are masked to zero weight, and their stale V rows are zeroed in shared memory before the
// P.V product.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "lg_common.cuh"
#include "lg_internal.h"

namespace lg {

namespace {

constexpr int kTile = 128;          // rows per tile (TMA box height)
constexpr int kBoxBytes = kTile * 128;  // one box: 128 rows x 64 bf16
constexpr int kConsumerWarps = 4;
constexpr int kProducerWarp = kConsumerWarps;
constexpr int kMergerWarp0 = kConsumerWarps + 1;
constexpr int kMergers = 4;   // merger warps; ticket k goes to merger k % kMergers
constexpr int kThreads = (kConsumerWarps + 1 + kMergers) * 32;
constexpr int kTickets = 2 * kMergers;  // finished chunks queued from the consumers to the mergers
                                        // (ticket k in slot k % kTickets, owned by merger k % 4)
constexpr int kMaxChunkRows = 4096;  // chunk rows at most (the tail of a call is about one chunk)
constexpr int kStagedSeqs = 256;     // lengths and offsets kept in shared memory up to this batch
constexpr int kL2KeepBytes = 32 << 20;  // K/V a short pass leaves in L2 at normal priority

template <int D>
struct MmaCfg {
  static constexpr int kHalves = D / 64;                      // boxes per row
  static constexpr int kStageBytes = 2 * kHalves * kBoxBytes;  // K and V
  static constexpr int kStages = D == 128 ? 3 : 6;
  static constexpr int kRingBytes = kStages * kStageBytes;
  // ticket buffers: room for one buffer of 8 heads; fewer heads fit more buffers
  static constexpr int kMergeBytes = kConsumerWarps * 8 * (D + 8) * 4;
  static constexpr int kQBytes = 8 * D * 2;  // a stage's query rows (up to 8 heads), bf16
  static constexpr int kSmem = kRingBytes + kMergeBytes + kStages * kQBytes + 1024;  // + slack
  static constexpr int kKSteps = D / 16;
};

// One ticket buffer: every consumer warp's chunk partial of the G real heads,
// o as [warp][head][D + 4] (the padding spreads the fragment stores over all banks), then
// {M, l, u, sigma} as [warp][head][4].
template <int D, int G>
struct TicketBuf {
  static constexpr int kOStride = D + 4;
  static constexpr int kFloats = kConsumerWarps * G * (kOStride + 4);
  static constexpr int kFit = MmaCfg<D>::kMergeBytes / (kFloats * 4);
  static constexpr int kBufs = kFit >= 8 ? 8 : (kFit >= 4 ? 4 : (kFit >= 2 ? 2 : 1));
  static_assert(kFit >= 1, "ticket buffer larger than its shared-memory budget");
};

// group arrival count: release (this chunk's partial, stored by the warp before) and acquire
// (the other chunks' partials, read by the arrival that completes the group) at GPU scope
__device__ __forceinline__ int arrive_acq_rel(int *p) {
  int old;
  asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], 1;" : "=r"(old) : "l"(p) : "memory");
  return old;
}

// 2-D tensor copy of one box into shared memory, completing on `bar`, with an L2 eviction
// policy (createpolicy) for the lines it brings in.
__device__ __forceinline__ void tma_load_2d(void *smem_dst, const CUtensorMap *map, int x,
                                                 int y, uint64_t *bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(smem_addr(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar)), "l"(policy)
      : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2,
                                        uint32_t &r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t &r0, uint32_t &r1,
                                              uint32_t &r2, uint32_t &r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

__device__ __forceinline__ void mma_bf16(float *d, uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, "
      "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(d) : "r"(a));
  return d;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}

// byte offset of 16-byte chunk c8 (0..7) of row r in a 128-byte-swizzled box
__device__ __forceinline__ uint32_t swz(int r, int c8) {
  return (uint32_t)(r * 128 + ((c8 ^ (r & 7)) << 4));
}

struct ChunkId {
  int lloc, b, kvh, ch;
};

// Chunk geometry of one call, from the lengths it attends over (the host sizes the workspace
// for max_len, which can be far above them): chunk rows a multiple of the tile, never more
// chunks per group than the workspace holds (max_chunks).  A CTA takes about one chunk per
// eight of its tiles, at least 3 (a chunk end costs the consumers a hand-off, and a short pass
// with fewer, longer chunks measured faster: at the paper-shaped step 2 chunks of 512 rows per
// group balance 152 CTAs better than 3 of 384) and at most 16 (measured: finer chunks gained
// nothing at the end of long passes and cost a little on the way); the rows are then evened
// out over the chunks of the longest group.
struct Geom {
  int rows;        // rows per chunk
  int per_grp;     // chunk ids per (layer, sequence, kv-head)
  int total;       // chunk ids of the call
  int groups;      // (layer, sequence, kv-head) groups of the call
  bool long_pass;  // the last chunks of the groups are short and claimed last; no reversal
};

__device__ __forceinline__ Geom make_geom(const AttendArgs &a, int n_max, int64_t len_sum,
                                          int ctas) {
  // the chunks per CTA and the rows they imply are a heuristic: float arithmetic (the same in
  // every CTA) keeps 64-bit divisions off the prologue
  const float rows_all = (float)len_sum * (float)(a.H_kv * a.n_layers);
  const float per_cta =
      fminf(fmaxf(floorf(rows_all / (float)(kTile * 8) / (float)ctas), 3.f), 16.f);
  const float cf = ceilf(rows_all / ((float)ctas * per_cta));
  int c = cf >= (float)kMaxChunkRows ? kMaxChunkRows : (int)cf;
  const unsigned nm = (unsigned)n_max;
  const int fit = (int)((nm + (unsigned)a.max_chunks - 1u) / (unsigned)a.max_chunks);
  c = max(max(c, fit), kTile);
  c = (c + kTile - 1) / kTile * kTile;
  // even rows: as many chunks per group, each about n_max / per_grp rows (no more chunks, so
  // still within max_chunks)
  const unsigned per = max(1u, (nm + (unsigned)c - 1u) / (unsigned)c);
  c = (int)(((nm + per - 1u) / per + kTile - 1) / kTile * kTile);
  c = max(c, kTile);
  Geom gm;
  // a long pass (64 tiles a CTA or more) ends on short chunks: each group's last chunk is
  // about an eighth of the others (rows n_max / (per - 7/8), as many chunks per group), and
  // decode_chunk hands out every group's last chunk after all the others (an eighth against a
  // quarter, same-box A/B: workload 2 +0.3 %, workloads 4 and 5 unchanged)
  gm.long_pass = rows_all >= 64.f * (float)kTile * (float)ctas && per >= 2;
  if (gm.long_pass) {
    const float cl = ceilf((float)nm / ((float)per - 0.875f));
    c = max(c, ((int)cl + kTile - 1) / kTile * kTile);
  }
  gm.rows = c;
  gm.per_grp = max(1, (int)((nm + (unsigned)c - 1u) / (unsigned)c));
  gm.groups = a.n_layers * a.batch * a.H_kv;
  gm.total = gm.groups * gm.per_grp;
  return gm;
}

// Chunk id -> (layer, sequence, kv-head, chunk): the groups' chunks but the last come first
// (per_grp - 1 of each group, group-major), then every group's last chunk.
__device__ __forceinline__ ChunkId decode_chunk(const AttendArgs &a, int c, const Geom &gm) {
  ChunkId id;
  const int nb = gm.per_grp - 1;
  int r;
  if (c < gm.groups * nb) {
    id.ch = c % nb;
    r = c / nb;
  } else {
    id.ch = nb;
    r = c - gm.groups * nb;
  }
  id.kvh = r % a.H_kv;
  r /= a.H_kv;
  id.b = r % a.batch;
  id.lloc = r / a.batch;
  return id;
}

// Split-K merge of one group's chunk partials (all G heads, one warp):
//   M = max_j M_j, f_j = 2^(M_j - M), l = sum f_j l_j, u = sum f_j (u_j + (M_j - M) l_j),
//   sigma = sum f_j sigma_j, o = sum f_j o_j / l
// out = o, stats = {M ln 2, l, ln l - u ln 2 / l, sigma / l}.  The partials were written by
// other CTAs of this launch: read through L2.  Lane j holds chunk j's {M, l, u, sigma} (up to
// 32 chunks; more are read again per block), and the o slices of up to eight chunks are loaded
// with them; heads go two at a time (an even G of 4 or more), so a group of at most eight
// chunks costs one round trip per pair of heads.
template <int D, int H>
__device__ __forceinline__ void merge_heads(const AttendArgs &a, int64_t head_first, int nch,
                                            int lane) {
  constexpr int EPL = D / 32;
  constexpr int kBlk = 8;
  const float *pp[H];
  float ob[H][kBlk][EPL];
  float4 sl[H];
#pragma unroll
  for (int hh = 0; hh < H; ++hh) {
    pp[hh] = a.partial + (head_first + hh) * a.max_chunks * (D + 8);
#pragma unroll
    for (int jj = 0; jj < kBlk; ++jj)
#pragma unroll
      for (int k = 0; k < EPL; ++k)
        ob[hh][jj][k] =
            jj < nch ? __ldcg(pp[hh] + (int64_t)jj * (D + 8) + 8 + lane + 32 * k) : 0.f;
    sl[hh] = make_float4(-INFINITY, 0.f, 0.f, 0.f);  // this lane's chunk (j = lane)
    if (lane < nch)
      sl[hh] = __ldcg(reinterpret_cast<const float4 *>(pp[hh] + (int64_t)lane * (D + 8)));
  }
  float M[H], l[H], u[H], sg[H], acc[H][EPL];
#pragma unroll
  for (int hh = 0; hh < H; ++hh) {
    M[hh] = sl[hh].x;
    for (int j = lane + 32; j < nch; j += 32)
      M[hh] = fmaxf(M[hh], __ldcg(pp[hh] + (int64_t)j * (D + 8)));
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) M[hh] = fmaxf(M[hh], __shfl_xor_sync(0xffffffffu, M[hh], o));
    l[hh] = u[hh] = sg[hh] = 0.f;
#pragma unroll
    for (int k = 0; k < EPL; ++k) acc[hh][k] = 0.f;
  }
  for (int j0 = 0; j0 < nch; j0 += kBlk) {
#pragma unroll
    for (int hh = 0; hh < H; ++hh) {
      if (j0 > 0) {
#pragma unroll
        for (int jj = 0; jj < kBlk; ++jj)
#pragma unroll
          for (int k = 0; k < EPL; ++k)
            ob[hh][jj][k] = j0 + jj < nch
                                ? __ldcg(pp[hh] + (int64_t)(j0 + jj) * (D + 8) + 8 + lane + 32 * k)
                                : 0.f;
      }
      // weights of this block's chunks: lane jj < kBlk takes chunk j0 + jj (held by lane
      // j0 + jj when that is below 32, read again otherwise)
      const int j = j0 + lane;
      float4 sv = make_float4(__shfl_sync(0xffffffffu, sl[hh].x, j & 31),
                              __shfl_sync(0xffffffffu, sl[hh].y, j & 31),
                              __shfl_sync(0xffffffffu, sl[hh].z, j & 31),
                              __shfl_sync(0xffffffffu, sl[hh].w, j & 31));
      float f = 0.f;
      if (lane < kBlk && j < nch) {
        if (j >= 32) sv = __ldcg(reinterpret_cast<const float4 *>(pp[hh] + (int64_t)j * (D + 8)));
        f = exp2f(sv.x - M[hh]);
        l[hh] += f * sv.y;
        u[hh] += f * (sv.z + (sv.x - M[hh]) * sv.y);
        sg[hh] += f * sv.w;
      }
#pragma unroll
      for (int jj = 0; jj < kBlk; ++jj) {
        const float fj = __shfl_sync(0xffffffffu, f, jj);
#pragma unroll
        for (int k = 0; k < EPL; ++k) acc[hh][k] += fj * ob[hh][jj][k];
      }
    }
  }
#pragma unroll
  for (int hh = 0; hh < H; ++hh) {
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) {
      l[hh] += __shfl_xor_sync(0xffffffffu, l[hh], o);
      u[hh] += __shfl_xor_sync(0xffffffffu, u[hh], o);
      sg[hh] += __shfl_xor_sync(0xffffffffu, sg[hh], o);
    }
    const int64_t head = head_first + hh;
    const float inv_l = 1.f / l[hh];
    __nv_bfloat16 *out = reinterpret_cast<__nv_bfloat16 *>(a.out) + head * D;
#pragma unroll
    for (int k = 0; k < EPL; ++k) out[lane + 32 * k] = __float2bfloat16_rn(acc[hh][k] * inv_l);
    if (lane == 0) {
      constexpr float kLn2 = 0.69314718055994530942f;
      float *st = a.stats + head * 4;
      st[0] = M[hh] * kLn2;
      st[1] = l[hh];
      st[2] = logf(l[hh]) - u[hh] * kLn2 * inv_l;
      st[3] = sg[hh] * inv_l;
      if (a.final_ml) {
        a.final_ml[head * 2] = M[hh];
        a.final_ml[head * 2 + 1] = l[hh];
      }
    }
  }
}

template <int D, int G>
__device__ __forceinline__ void merge_group(const AttendArgs &a, int64_t head0, int n,
                                            int chunk_rows, int lane) {
  const int nch = (n + chunk_rows - 1) / chunk_rows;
  // pairs of heads for an even G of 4 or more (measured: at G = 2 the pair is slower)
  constexpr int H = G % 2 == 0 && G >= 4 ? 2 : 1;
#pragma unroll 1
  for (int h = 0; h < G; h += H) merge_heads<D, H>(a, head0 + h, nch, lane);
}

}  // namespace

template <int D, int G>
__global__ void __launch_bounds__(kThreads, 1)
attend_mma_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                  AttendArgs a, int *next_chunk) {
  using C = MmaCfg<D>;
  extern __shared__ unsigned char smem_raw[];
  __shared__ __align__(8) uint64_t full_bar[C::kStages];
  __shared__ __align__(8) uint64_t empty_bar[C::kStages];
  __shared__ int stage_chunk[C::kStages];  // chunk of the tile in each stage, -1: no more work
  __shared__ int stage_tile[C::kStages];   // tile index within that chunk
  __shared__ int stage_n[C::kStages];      // the chunk's sequence length
  __shared__ long long stage_lrow0[C::kStages];  // its first row in the logits layout
  using TB = TicketBuf<D, G>;
  __shared__ __align__(8) uint64_t tfull[kTickets];   // consumers -> merger: a finished chunk
  __shared__ __align__(8) uint64_t tempty[kTickets];  // merger -> consumers: the slot is free
  __shared__ __align__(8) uint64_t bfree[TB::kBufs];  // merger -> consumers: the buffer is read
  __shared__ int t_grp[kTickets], t_n[kTickets], t_ch[kTickets];  // group (-1: no more), length,
                                                                   // chunk within the group
  __shared__ int red_max[kThreads / 32];
  __shared__ long long red_sum[kThreads / 32];
  __shared__ int s_len[kStagedSeqs];         // len[b] and seq_off[b] of a batch up to kStagedSeqs
  __shared__ long long s_off[kStagedSeqs];
  __shared__ int s_bad;                      // the device status at entry (one read per CTA)
  __shared__ int s_rev;                      // this call walks its chunks from the last one
  unsigned char *smem = reinterpret_cast<unsigned char *>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  float *tbuf = reinterpret_cast<float *>(smem + C::kRingBytes);  // [kBufs][TB::kFloats]
  unsigned char *qbuf = smem + C::kRingBytes + C::kMergeBytes;      // [stages][8][D] bf16

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // CTA i starts on chunk i; later chunks come from the shared counter (offset by the grid)
  if (warp == kProducerWarp && lane == 0) {
    // the descriptors' fetch overlaps the prologue
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
  }
  pdl_enter();  // the tensormap prefetch above reads only the kernel's parameters
  if (threadIdx.x == 0) {
    s_bad = status_bad(a.status);
    s_rev = a.counter[1 + a.n_layers * a.batch * a.H_kv] & 1;
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], kConsumerWarps);
    }
    for (int s = 0; s < kTickets; ++s) {
      mbar_init(&tfull[s], kConsumerWarps);
      mbar_init(&tempty[s], 1);
    }
    for (int s = 0; s < TB::kBufs; ++s) mbar_init(&bfree[s], 1);
    mbar_fence_init();
  }
  {
    // longest and total length of the batch (lengths past max_len count as max_len)
    int nmx = 0;
    long long sum = 0;
    for (int b = threadIdx.x; b < a.batch; b += kThreads) {
      const int nb = a.len[b];
      if (b < kStagedSeqs) {
        s_len[b] = nb;
        s_off[b] = a.seq_off[b];
      }
      const int n = min(nb, a.max_len);
      nmx = max(nmx, n);
      sum += n;
    }
    nmx = __reduce_max_sync(0xffffffffu, nmx);
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    if (lane == 0) {
      red_max[warp] = nmx;
      red_sum[warp] = sum;
    }
  }
  __syncthreads();
  if (s_bad) return;  // the same decision in every thread of the CTA
  const bool staged = a.batch <= kStagedSeqs;
  int n_max = 0;
  long long len_sum = 0;
#pragma unroll
  for (int w = 0; w < kThreads / 32; ++w) {
    n_max = max(n_max, red_max[w]);
    len_sum += red_sum[w];
  }
  const Geom gm = make_geom(a, n_max, len_sum, gridDim.x);

  if (warp >= kMergerWarp0) {
    // ------------------------------------------------------------ mergers
    // One ticket per finished chunk, dealt round-robin to the merger warps; ticket k's warp
    // partials are in buffer k % kBufs.  The merger folds the four into the chunk's partial
    // {M, l, u, sigma, o} (global, read by the group's last arrival), frees the buffer, and
    // counts the arrival.  The consumers' buffer stores are ordered before the ticket (each
    // warp's __syncwarp and mbarrier release, the merger's acquire); the arrival count is an
    // acquire-release atomic at GPU scope after the warp's __syncwarp, so the chunk partial is
    // visible before the count moves, and the arrival that completes the group reads every
    // chunk partial of the group.
    for (uint32_t tk = warp - kMergerWarp0;; tk += kMergers) {
      const int slot = tk % kTickets;
      if (!mbar_wait(&tfull[slot], (tk / kTickets) & 1)) {
        set_status(a.status, LG_ERR_TIMEOUT);
        return;
      }
      const int grp = t_grp[slot], n = t_n[slot], ch = t_ch[slot];
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[slot]);
      if (grp < 0) break;
      const int64_t head0 = (int64_t)(grp / a.H_kv) * a.H_q + (int64_t)(grp % a.H_kv) * G;
      {
        const float *ob = tbuf + (size_t)(tk % TB::kBufs) * TB::kFloats;
        const float *sb = ob + kConsumerWarps * G * TB::kOStride;
#pragma unroll 1
        for (int h = 0; h < G; ++h) {
          float4 ws[kConsumerWarps];
          float M = -INFINITY;
#pragma unroll
          for (int w = 0; w < kConsumerWarps; ++w) {
            ws[w] = *reinterpret_cast<const float4 *>(sb + (w * G + h) * 4);
            M = fmaxf(M, ws[w].x);
          }
          float f[kConsumerWarps], l = 0.f, u = 0.f, sg = 0.f;
#pragma unroll
          for (int w = 0; w < kConsumerWarps; ++w) {
            // a warp that saw no row of this chunk has l = 0, M = -inf and no weight
            f[w] = 0.f;
            if (ws[w].y > 0.f) {
              f[w] = exp2f(ws[w].x - M);
              l += f[w] * ws[w].y;
              u += f[w] * (ws[w].z + (ws[w].x - M) * ws[w].y);
              sg += f[w] * ws[w].w;
            }
          }
          float *pp = a.partial + ((head0 + h) * a.max_chunks + ch) * (D + 8);
#pragma unroll
          for (int k = 0; k < D / 32; ++k) {
            const int e = lane + 32 * k;
            float ov = 0.f;
#pragma unroll
            for (int w = 0; w < kConsumerWarps; ++w)
              ov += f[w] * ob[(w * G + h) * TB::kOStride + e];
            pp[8 + e] = ov;
          }
          if (lane == 0) *reinterpret_cast<float4 *>(pp) = make_float4(M, l, u, sg);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&bfree[tk % TB::kBufs]);
      int last = 0;
      if (lane == 0) {
        const int nch = (n + gm.rows - 1) / gm.rows;
        last = arrive_acq_rel(a.counter + 1 + grp) == nch - 1;
      }
      last = __shfl_sync(0xffffffffu, last, 0);
      __syncwarp();  // the lanes' partial reads follow lane 0's acquire
      if (last) {
        merge_group<D, G>(a, head0, n, gm.rows, lane);
      }
    }
    return;
  }

  if (warp == kProducerWarp) {
    // ------------------------------------------------------------ producer
    // A CTA's first two chunks are blockIdx.x and blockIdx.x + gridDim.x; later ones come from
    // a shared counter (ragged lengths balance across CTAs), each claimed as its predecessor
    // starts (one ahead: the claim's round trip overlaps a chunk, and a CTA near the end of the
    // pass holds at most one chunk it has not started); each stage carries its chunk,
    // tile index, length and logits row to the consumers, and a chunk's first stage also
    // brings the chunk's query rows (one bulk copy on the same barrier).
    if (lane == 0) {
      // K/V tiles are streamed once per call: their L2 lines go first when space is needed, so
      // that a pass of the whole cache does not evict what the rest of the step works on (the
      // other kernels' code and data, the workspace).  Same-box A/B at one sequence (115 MB of
      // K/V a step, less than the 129 MB L2; bench.py --workload 6): 41.7 -> 39.4 us per step,
      // the loop-onset test's share most of all.
      uint64_t evict_first, evict_normal;
      asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(evict_first));
      asm volatile("createpolicy.fractional.L2::evict_normal.b64 %0, 1.0;" : "=l"(evict_normal));
      // Except the chunks a short pass claims last, about kL2KeepBytes of them: the next call
      // walks the chunks the other way and starts on these, so they keep normal priority (its
      // first tiles came from DRAM otherwise: same-box A/B 35.4 -> 34.2 us per step).
      const int chunk_bytes = gm.rows * 4 * D;  // K and V rows of a full chunk
      const int keep_from =
          gm.long_pass ? gm.total : gm.total - max(1, (int)(kL2KeepBytes / chunk_bytes));
      uint32_t it = 0;
      const int claimed0 = 2 * (int)gridDim.x;
      const bool rev = s_rev != 0;
      int c = blockIdx.x;
      bool first = true;
      while (true) {
        const bool alive = c < gm.total;
        // the chunk this claim stands for: a short pass walks the chunks from the last on
        // every other call, so that it starts on the rows the previous call read last (still
        // in L2); a long pass keeps its order (its short last chunks stay at the end)
        const int cm = rev && !gm.long_pass ? gm.total - 1 - c : c;
        int ntiles = 0, grow = 0, n = 0, c_next = 0;
        int64_t lrow0 = 0, head0 = 0;
        uint64_t policy = evict_first;
        if (alive) {
          c_next = first ? (int)(blockIdx.x + gridDim.x) : claimed0 + atomicAdd(next_chunk, 1);
          first = false;
          const ChunkId id = decode_chunk(a, cm, gm);
          policy = c >= keep_from ? evict_normal : evict_first;
          n = staged ? s_len[id.b] : a.len[id.b];
          const int64_t off = staged ? s_off[id.b] : a.seq_off[id.b];
          const int row0 = id.ch * gm.rows;
          head0 = ((int64_t)id.lloc * a.batch + id.b) * a.H_q + (int64_t)id.kvh * G;
          if (n > a.max_len) set_status(a.status, LG_ERR_CAPACITY);
          if (n == 0 && id.ch == 0) {
            // empty sequence: no chunk to merge; zero output, m = -inf, l = H = S = 0
            __nv_bfloat16 *out = reinterpret_cast<__nv_bfloat16 *>(a.out) + head0 * D;
            for (int e = 0; e < G * D; ++e) out[e] = __float2bfloat16_rn(0.f);
            for (int h = 0; h < G; ++h) {
              a.stats[(head0 + h) * 4] = -INFINITY;
              a.stats[(head0 + h) * 4 + 1] = a.stats[(head0 + h) * 4 + 2] =
                  a.stats[(head0 + h) * 4 + 3] = 0.f;
            }
          }
          if (n > a.max_len || row0 >= n) {
            c = c_next;
            continue;
          }
          ntiles = (min(gm.rows, n - row0) + kTile - 1) / kTile;
          grow = (int)(((int64_t)(a.layer0 + id.lloc) * a.H_kv + id.kvh) * a.S_total + off + row0);
          lrow0 = ((int64_t)id.lloc * a.H_kv + id.kvh) * a.S_total + off + row0;
        }
        for (int t = 0; t < (alive ? ntiles : 1); ++t, ++it) {
          const int st = it % C::kStages;
          if (it >= (uint32_t)C::kStages &&
              !mbar_wait(&empty_bar[st], ((it / C::kStages) - 1) & 1)) {
            set_status(a.status, LG_ERR_TIMEOUT);
            return;
          }
          stage_chunk[st] = alive ? cm : -1;
          stage_tile[st] = t;
          stage_n[st] = n;
          stage_lrow0[st] = lrow0;
          if (!alive) {
            mbar_arrive(&full_bar[st]);  // end of work: completes the phase without a copy
            break;
          }
          unsigned char *stage = smem + (size_t)st * C::kStageBytes;
          mbar_arrive_expect_tx(&full_bar[st], C::kStageBytes + (t == 0 ? G * D * 2 : 0));
#pragma unroll
          for (int h = 0; h < C::kHalves; ++h) {
            tma_load_2d(stage + h * kBoxBytes, &tmK, h * 64, grow + t * kTile,
                             &full_bar[st], policy);
            tma_load_2d(stage + (C::kHalves + h) * kBoxBytes, &tmV, h * 64,
                             grow + t * kTile, &full_bar[st], policy);
          }
          if (t == 0)
            bulk_load(qbuf + st * C::kQBytes,
                      reinterpret_cast<const __nv_bfloat16 *>(a.q) + head0 * D, G * D * 2,
                      &full_bar[st]);
        }
        if (!alive) break;
        c = c_next;
      }
    }
    return;
  }

  // -------------------------------------------------------------- consumers
  const int g = lane >> 2, t4 = lane & 3;
  const int mrow = lane & 7, msel = lane >> 3;  // ldmatrix: row within 8x8, matrix index
  ChunkId id;
  int n = 0, row0 = 0, rows = 0, ntiles = 0, suffix_lo = 0;
  int64_t lrow0 = 0;
  uint32_t qf[C::kKSteps][2];
  float o[C::kKSteps][4];
  float m2[2], l2[2], u2[2], sg2[2];
  float *logits = a.logits;
  uint32_t tk = 0;        // tickets issued (the same count in every consumer warp)
  bool handoff = true;    // false once a buffer or ticket slot was not released in time
  for (uint32_t it = 0;; ++it) {
    const int st = it % C::kStages;
    if (!mbar_wait(&full_bar[st], (it / C::kStages) & 1)) {
      set_status(a.status, LG_ERR_TIMEOUT);
      return;
    }
    const int c = stage_chunk[st];
    if (c < 0) break;
    const int t = stage_tile[st];
    if (t == 0) {
      // first tile of a chunk: its geometry, the q^T fragments, fresh softmax state
      id = decode_chunk(a, c, gm);
      n = stage_n[st];
      row0 = id.ch * gm.rows;
      rows = min(gm.rows, n - row0);
      ntiles = (rows + kTile - 1) / kTile;
      suffix_lo = n - min(a.suffix_w, n);
      lrow0 = stage_lrow0[st];
      // B fragments of q^T: head g (zero for padded heads), d = 16 ks + 2 t4 (+1, +8, +9)
      const uint32_t *qp = reinterpret_cast<const uint32_t *>(qbuf + st * C::kQBytes) + g * (D / 2);
#pragma unroll
      for (int ks = 0; ks < C::kKSteps; ++ks) {
        qf[ks][0] = g < G ? qp[ks * 8 + t4] : 0u;
        qf[ks][1] = g < G ? qp[ks * 8 + 4 + t4] : 0u;
      }
#pragma unroll
      for (int eb = 0; eb < C::kKSteps; ++eb) o[eb][0] = o[eb][1] = o[eb][2] = o[eb][3] = 0.f;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        m2[h] = -INFINITY;
        l2[h] = u2[h] = sg2[h] = 0.f;
      }
    }
    unsigned char *stage = smem + (size_t)st * C::kStageBytes;
    const uint32_t kbase = smem_addr(stage);
    const uint32_t vbase = kbase + C::kHalves * kBoxBytes;
    const int tile_rows = min(kTile, rows - t * kTile);
    const int r_w = warp * 32;  // this warp's first row in the tile
    if (tile_rows < r_w + 32) {
      // ragged tail: zero the V rows past the end so that 0 * stale stays 0
      for (int idx = lane; idx < 32 * C::kHalves * 8; idx += 32) {
        const int rr = r_w + idx / (C::kHalves * 8);
        const int hc = idx % (C::kHalves * 8);
        if (rr >= tile_rows)
          *reinterpret_cast<uint4 *>(stage + (C::kHalves + hc / 8) * kBoxBytes + rr * 128 +
                                     (hc % 8) * 16) = make_uint4(0u, 0u, 0u, 0u);
      }
      __syncwarp();
    }

    // S^T for the warp's two 16-row blocks
    float s[2][4];
#pragma unroll
    for (int mb = 0; mb < 2; ++mb) {
      s[mb][0] = s[mb][1] = s[mb][2] = s[mb][3] = 0.f;
      const int r = r_w + mb * 16 + (msel & 1) * 8 + mrow;
#pragma unroll
      for (int ks = 0; ks < C::kKSteps; ++ks) {
        const int c8 = (ks & 3) * 2 + (msel >> 1);
        uint32_t a0, a1, a2, a3;
        ldsm_x4(kbase + (ks >> 2) * kBoxBytes + swz(r, c8), a0, a1, a2, a3);
        mma_bf16(s[mb], a0, a1, a2, a3, qf[ks][0], qf[ks][1]);
      }
    }
    // scale to log2 units, mask rows past the end; tile max per head (heads 2 t4, 2 t4 + 1)
    float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
    for (int mb = 0; mb < 2; ++mb)
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int rl = r_w + mb * 16 + g + (j >> 1) * 8;  // row within the tile
        const bool valid = rl < tile_rows;
        s[mb][j] = valid ? s[mb][j] * a.qscale : -INFINITY;
        mx[j & 1] = fmaxf(mx[j & 1], s[mb][j]);
      }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 4));
      mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 8));
      mx[h] = fmaxf(mx[h], __shfl_xor_sync(0xffffffffu, mx[h], 16));
    }
    const bool raise = mx[0] > m2[0] || mx[1] > m2[1];
    if (__any_sync(0xffffffffu, raise)) {
      float corr[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const float mn = fmaxf(m2[h], mx[h]);
        corr[h] = mn == m2[h] ? 1.f : exp2f(m2[h] - mn);
        u2[h] = l2[h] > 0.f ? corr[h] * (u2[h] + (m2[h] - mn) * l2[h]) : 0.f;
        l2[h] *= corr[h];
        sg2[h] *= corr[h];
        m2[h] = mn;
      }
#pragma unroll
      for (int eb = 0; eb < C::kKSteps; ++eb) {
        o[eb][0] *= corr[0];
        o[eb][1] *= corr[1];
        o[eb][2] *= corr[0];
        o[eb][3] *= corr[1];
      }
    }
    // probabilities, sums, and P^T fragments
    uint32_t pb[2][2], pl[2][2];
#pragma unroll
    for (int mb = 0; mb < 2; ++mb) {
      float p[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int h = j & 1;
        const int rl = r_w + mb * 16 + g + (j >> 1) * 8;
        const bool valid = rl < tile_rows;
        p[j] = valid ? exp2f(s[mb][j] - m2[h]) : 0.f;
        if (valid) {
          l2[h] += p[j];
          u2[h] += p[j] * (s[mb][j] - m2[h]);
          if (row0 + t * kTile + rl >= suffix_lo) sg2[h] += p[j];
        }
      }
      if (logits) {
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          const int rl = r_w + mb * 16 + g + half * 8;
          if (rl < tile_rows) {
            float *dst = logits + (lrow0 + t * kTile + rl) * G;
            if (G % 2 == 0) {
              // heads 2 t4 and 2 t4 + 1 side by side: one 8-byte store (rows of an even G
              // start 8-byte aligned)
              if (2 * t4 < G)
                *reinterpret_cast<float2 *>(dst + 2 * t4) =
                    make_float2(s[mb][half * 2], s[mb][half * 2 + 1]);
            } else {
              if (2 * t4 < G) dst[2 * t4] = s[mb][half * 2];
              if (2 * t4 + 1 < G) dst[2 * t4 + 1] = s[mb][half * 2 + 1];
            }
          }
        }
      }
      // P = hi + lo, both bf16: the P.V product keeps ~16 mantissa bits of P
      const uint32_t h01 = pack_bf16(p[0], p[1]), h23 = pack_bf16(p[2], p[3]);
      const float2 f01 = bf16x2_to_float2(h01), f23 = bf16x2_to_float2(h23);
      pb[mb][0] = movmatrix_trans(h01);  // rows 0-7 of the block
      pb[mb][1] = movmatrix_trans(h23);  // rows 8-15
      pl[mb][0] = movmatrix_trans(pack_bf16(p[0] - f01.x, p[1] - f01.y));
      pl[mb][1] = movmatrix_trans(pack_bf16(p[2] - f23.x, p[3] - f23.y));
    }
    // o^T += V^T P^T
#pragma unroll
    for (int mb = 0; mb < 2; ++mb) {
      const int r = r_w + mb * 16 + (msel >> 1) * 8 + mrow;
#pragma unroll
      for (int eb = 0; eb < C::kKSteps; ++eb) {
        const int c8 = (eb & 3) * 2 + (msel & 1);
        uint32_t a0, a1, a2, a3;
        ldsm_x4_trans(vbase + (eb >> 2) * kBoxBytes + swz(r, c8), a0, a1, a2, a3);
        mma_bf16(o[eb], a0, a1, a2, a3, pb[mb][0], pb[mb][1]);
        mma_bf16(o[eb], a0, a1, a2, a3, pl[mb][0], pl[mb][1]);
      }
    }
    __syncwarp();
    if (tile_rows < r_w + 32) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    if (lane == 0) mbar_arrive(&empty_bar[st]);
    if (t != ntiles - 1) continue;

    // ---------------------------------------------------------- chunk done: hand it off
    // This warp's sums over its rows (lanes of one t4 hold the rows g, g + 8 of a head pair).
#pragma unroll
    for (int h = 0; h < 2; ++h) {
#pragma unroll
      for (int off = 4; off <= 16; off <<= 1) {
        l2[h] += __shfl_xor_sync(0xffffffffu, l2[h], off);
        u2[h] += __shfl_xor_sync(0xffffffffu, u2[h], off);
        sg2[h] += __shfl_xor_sync(0xffffffffu, sg2[h], off);
      }
    }
    if (!handoff) continue;
    const int buf = tk % TB::kBufs, slot = tk % kTickets;
    int ok = 1;
    if (lane == 0) {
      // the buffer's previous ticket has been read by its merger (so every warp has arrived on
      // every ticket up to kBufs <= kTickets back, and this arrival counts toward this ticket);
      // warp 0 also waits for the ticket slot before writing its group, length and chunk
      if (tk >= (uint32_t)TB::kBufs && !mbar_wait(&bfree[buf], ((tk / TB::kBufs) - 1) & 1))
        ok = 0;
      if (ok && warp == 0) {
        if (tk >= (uint32_t)kTickets && !mbar_wait(&tempty[slot], ((tk / kTickets) - 1) & 1)) {
          ok = 0;
        } else {
          t_grp[slot] = (int)(((int64_t)id.lloc * a.batch + id.b) * a.H_kv + id.kvh);
          t_n[slot] = n;
          t_ch[slot] = id.ch;
        }
      }
      if (!ok) set_status(a.status, LG_ERR_TIMEOUT);
    }
    if (!__shfl_sync(0xffffffffu, ok, 0)) {
      handoff = false;
      continue;
    }
    __syncwarp();  // the lanes' stores below follow lane 0's wait
    {
      // o^T fragments: this thread holds o[e][2 t4 + h2] for e = 16 eb + g (+8)
      float *ob = tbuf + (size_t)buf * TB::kFloats + warp * G * TB::kOStride;
      float *sb =
          tbuf + (size_t)buf * TB::kFloats + kConsumerWarps * G * TB::kOStride + warp * G * 4;
#pragma unroll
      for (int h2 = 0; h2 < 2; ++h2) {
        const int h = 2 * t4 + h2;
        if (h < G) {
#pragma unroll
          for (int eb = 0; eb < C::kKSteps; ++eb) {
            ob[h * TB::kOStride + eb * 16 + g] = o[eb][h2];
            ob[h * TB::kOStride + eb * 16 + g + 8] = o[eb][h2 + 2];
          }
          if (g == 0)
            *reinterpret_cast<float4 *>(sb + h * 4) = make_float4(m2[h2], l2[h2], u2[h2], sg2[h2]);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&tfull[slot]);
    ++tk;
  }
  if (handoff && lane == 0) {
    // no more chunks: one last ticket for each merger (no buffer).  Every warp first waits for
    // the slot's previous ticket to be taken, so that its arrival cannot count toward a ticket
    // another warp has not finished (end tickets follow no buffer wait)
    for (int m = 0; m < kMergers; ++m, ++tk) {
      const int slot = tk % kTickets;
      if (tk >= (uint32_t)kTickets && !mbar_wait(&tempty[slot], ((tk / kTickets) - 1) & 1)) {
        set_status(a.status, LG_ERR_TIMEOUT);
        break;
      }
      if (warp == 0) {
        t_grp[slot] = -1;
        t_n[slot] = 0;
        t_ch[slot] = 0;
      }
      mbar_arrive(&tfull[slot]);
    }
  }
}

// The call's chunk and group counters to zero (a kernel rather than a memset, so that the pass
// after it keeps its programmatic launch edge), and the word after them flipped: its low bit
// is the direction of this call's pass (any start value will do; it only alternates).
__global__ void zero_counters_kernel(int *p, int n) {
  pdl_enter();
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < n; i += gridDim.x * blockDim.x) p[i] = 0;
  if (blockIdx.x == 0 && threadIdx.x == 0) p[n] ^= 1;
}

// ------------------------------------------------------------------ host side

namespace {

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
      p = nullptr;
    return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }();
  return fn;
}

// 2-D view [L * H_kv * S_total rows][d] of one cache tensor, boxes of 128 rows x 64 columns
bool make_map(CUtensorMap *m, const void *base, int d, int64_t rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)d * 2};
  cuuint32_t box[2] = {64, (cuuint32_t)kTile};
  cuuint32_t estr[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D, int G>
cudaError_t launch_mma_typed(const CUtensorMap &mk, const CUtensorMap &mv, const AttendArgs &a,
                             int grid, int *counter, cudaStream_t s) {
  auto kern = attend_mma_kernel<D, G>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, MmaCfg<D>::kSmem);
  if (e != cudaSuccess) return e;
  LG_TRY(launch_pdl(kern, grid, kThreads, MmaCfg<D>::kSmem, s, mk, mv, a, counter));
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_mma_d(const CUtensorMap &mk, const CUtensorMap &mv, const AttendArgs &a, int g,
                         int grid, int *counter, cudaStream_t s) {
  switch (g) {
    case 1: return launch_mma_typed<D, 1>(mk, mv, a, grid, counter, s);
    case 2: return launch_mma_typed<D, 2>(mk, mv, a, grid, counter, s);
    case 3: return launch_mma_typed<D, 3>(mk, mv, a, grid, counter, s);
    case 4: return launch_mma_typed<D, 4>(mk, mv, a, grid, counter, s);
    case 5: return launch_mma_typed<D, 5>(mk, mv, a, grid, counter, s);
    case 6: return launch_mma_typed<D, 6>(mk, mv, a, grid, counter, s);
    case 7: return launch_mma_typed<D, 7>(mk, mv, a, grid, counter, s);
    case 8: return launch_mma_typed<D, 8>(mk, mv, a, grid, counter, s);
  }
  return cudaErrorInvalidValue;
}

}  // namespace

int mma_tile_rows() { return kTile; }

cudaError_t launch_attend_mma_partial(const AttendArgs &a, int d, int g, int64_t rows_total,
                                      cudaStream_t s) {
  CUtensorMap mk, mv;
  if (!make_map(&mk, a.K, d, rows_total) || !make_map(&mv, a.V, d, rows_total))
    return cudaErrorInvalidValue;
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return e;
  // an upper bound of the chunk ids (the kernel sizes its chunks from the lengths it reads)
  const int total = a.n_layers * a.batch * a.H_kv * a.max_chunks;
  const int grid = total < sms ? total : sms;
  if (!a.counter) return cudaErrorInvalidValue;
  const size_t counters = (size_t)(1 + (int64_t)a.n_layers * a.batch * a.H_kv) * sizeof(int);
  {
    const int n = (int)(counters / sizeof(int));
    const int blocks = (n + 255) / 256 < sms ? (n + 255) / 256 : sms;
    if ((e = launch_pdl(zero_counters_kernel, blocks, 256, 0, s, a.counter, n)) != cudaSuccess)
      return e;
  }
  if (d == 128) return launch_mma_d<128>(mk, mv, a, g, grid, a.counter, s);
  if (d == 64) return launch_mma_d<64>(mk, mv, a, g, grid, a.counter, s);
  return cudaErrorInvalidValue;
}

}  // namespace lg
