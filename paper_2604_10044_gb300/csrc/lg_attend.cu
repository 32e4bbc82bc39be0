// Split-K decode attention over the KV cache fused with the guard's per-head statistics
// (LoopGuard Sec. 3.1, Eq. 1; statistics read by Sec. 5.2), plus the H2O score accumulation
// of the comparator policy (Sec. 2.2, Sec. 6.1).
//
// One CTA streams CH consecutive rows of one (layer, sequence, kv-head) and serves all g query
// heads of that kv-head, so every K/V byte is read from HBM once per step.  A producer warp
// moves 8 KB K and V tiles into a 4-stage shared-memory ring with 1-D bulk copies (TMA)
// completing on mbarriers; four consumer warps compute.  A row is split over LPR lanes
// (16 B each): the lanes form partial dot products for all heads with packed fp32 FMAs, a
// transposed butterfly leaves each lane with the full logit of one head, that lane runs the
// online softmax for its head (in log2 units) and the probabilities are broadcast back for
// the P.V update.  The CTA writes one partial {M, l, u, sigma, o[d]} per head; a second kernel
// merges the partials of a head and emits out and the statistics {m, l, H, S}.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

#include "lg_common.cuh"
#include "lg_internal.h"

namespace lg {

template <typename T, int D, int G>
struct AttendCfg {
  static constexpr int kRowBytes = D * Elem<T>::kSize;  // 128, 256 or 512
  static constexpr int kLPR = kRowBytes / 16;           // lanes per row
  static constexpr int kEPL = 16 / Elem<T>::kSize;      // elements per lane
  static constexpr int kRPW = 32 / kLPR;                // rows per warp-step
  static constexpr int kGP = pow2_ceil(G);              // group padded to a power of two
  static constexpr int kWarps = 4;                      // consumer warps
  static constexpr int kThreads = (kWarps + 1) * 32;    // + one producer warp
  static constexpr int kTileBytes = 8192;               // per tensor per stage
  static constexpr int kTile = kTileBytes / kRowBytes;  // rows per stage
  static constexpr int kStages = 4;
  static constexpr int kRowsPerWarp = kTile / kWarps;
  static constexpr int kSteps = kRowsPerWarp / kRPW;    // warp-steps per stage
  static constexpr int kGroups = kWarps * kRPW;         // row groups per CTA
  static constexpr int kSmem = kStages * 2 * kTileBytes;
  static_assert(kGP <= kLPR, "GQA group wider than the lanes of a row");
  static_assert(kSteps >= 1, "tile too small");
  static_assert(kGroups * G * D * 4 + kGroups * kGP * 16 <= kSmem, "combine scratch");
};

// Leaves in v[0] the sum over the LPR lanes of a row of the partials of head
// lane_in_row / (LPR / GP): halving levels first (each lane keeps half of its heads and sends
// the other half to its partner), plain butterfly levels after.
template <int CNT, int OFF>
struct HeadReduce {
  __device__ __forceinline__ static void run(float *v, int lane) {
    if constexpr (CNT > 1) {
      constexpr int H = CNT / 2;
      const bool upper = (lane & OFF) != 0;
#pragma unroll
      for (int i = 0; i < H; ++i) {
        const float send = upper ? v[i] : v[i + H];
        const float keep = upper ? v[i + H] : v[i];
        v[i] = keep + __shfl_xor_sync(0xffffffffu, send, OFF);
      }
      HeadReduce<H, OFF / 2>::run(v, lane);
    } else if constexpr (OFF >= 1) {
      v[0] += __shfl_xor_sync(0xffffffffu, v[0], OFF);
      HeadReduce<1, OFF / 2>::run(v, lane);
    }
  }
};

__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) { return __ffma2_rn(a, b, c); }

template <typename T, int D, int G>
__global__ void __launch_bounds__(AttendCfg<T, D, G>::kThreads)
attend_partial_kernel(AttendArgs a) {
  pdl_enter();
  using C = AttendCfg<T, D, G>;
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ __align__(8) uint64_t full_bar[C::kStages];
  __shared__ __align__(8) uint64_t empty_bar[C::kStages];

  const int chunk = blockIdx.x, kvh = blockIdx.y;
  const int b = blockIdx.z % a.batch, lloc = blockIdx.z / a.batch;
  const int layer = a.layer0 + lloc;
  if (cta_status_bad(a.status)) return;
  const int n = a.len[b];
  if (n > a.max_len || n < 0) {
    if (threadIdx.x == 0) set_status(a.status, LG_ERR_CAPACITY);
    return;
  }
  const int row0 = chunk * a.chunk_rows;
  if (row0 >= n) return;
  const int rows = min(a.chunk_rows, n - row0);
  const int ntiles = (rows + C::kTile - 1) / C::kTile;
  const int64_t srow0 = ((int64_t)layer * a.H_kv + kvh) * a.S_total + a.seq_off[b] + row0;
  const unsigned char *Kg = (const unsigned char *)a.K + srow0 * C::kRowBytes;
  const unsigned char *Vg = (const unsigned char *)a.V + srow0 * C::kRowBytes;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&full_bar[s], 1);
      mbar_init(&empty_bar[s], C::kWarps);
    }
    mbar_fence_init();
  }
  __syncthreads();

  if (warp == C::kWarps) {
    // producer: one thread issues the bulk copies of every tile of the chunk
    if (lane == 0) {
      for (int t = 0; t < ntiles; ++t) {
        const int st = t % C::kStages;
        if (t >= C::kStages && !mbar_wait(&empty_bar[st], ((t / C::kStages) - 1) & 1)) {
          set_status(a.status, LG_ERR_TIMEOUT);
          break;
        }
        const int rt = min(C::kTile, rows - t * C::kTile);
        const uint32_t bytes = (uint32_t)rt * C::kRowBytes;
        unsigned char *ks = smem + (size_t)st * 2 * C::kTileBytes;
        mbar_arrive_expect_tx(&full_bar[st], 2 * bytes);
        bulk_load(ks, Kg + (size_t)t * C::kTileBytes, bytes, &full_bar[st]);
        bulk_load(ks + C::kTileBytes, Vg + (size_t)t * C::kTileBytes, bytes, &full_bar[st]);
      }
    }
    return;
  }

  // ---------------------------------------------------------------- consumers
  constexpr int LPR = C::kLPR, EPL = C::kEPL, GP = C::kGP, NP = EPL / 2;
  constexpr int DUP = LPR / GP;  // lanes holding the same head after the reduction
  const int li = lane % LPR;     // lane within its row
  const int gbase = lane - li;   // first lane of the row group
  const int hd = li / DUP;       // head this lane owns after the reduction
  const bool own = hd < G;
  const int rgrp = warp * C::kRPW + lane / LPR;  // row group id within the CTA

  // query slice of every head, prescaled by scale * log2(e)
  float2 q2[G][NP];
  {
    const int64_t qh0 = ((int64_t)lloc * a.batch + b) * a.H_q + (int64_t)kvh * G;
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const uint4 u = *reinterpret_cast<const uint4 *>(
          (const unsigned char *)a.q + ((qh0 + g) * D + li * EPL) * Elem<T>::kSize);
      float2 f[NP];
      Elem<T>::unpack(u, f);
#pragma unroll
      for (int j = 0; j < NP; ++j) q2[g][j] = make_float2(f[j].x * a.qscale, f[j].y * a.qscale);
    }
  }
  float2 o2[G][NP];
#pragma unroll
  for (int g = 0; g < G; ++g)
#pragma unroll
    for (int j = 0; j < NP; ++j) o2[g][j] = make_float2(0.f, 0.f);
  float m_ref = -INFINITY, l_acc = 0.f, u_acc = 0.f, sig = 0.f;
  const int suffix_lo = n - min(a.suffix_w, n);
  float *logits = a.logits;
  const int64_t lrow0 = ((int64_t)lloc * a.H_kv + kvh) * a.S_total + a.seq_off[b] + row0;
  bool ok = true;

  for (int t = 0; t < ntiles && ok; ++t) {
    const int st = t % C::kStages;
    if (!mbar_wait(&full_bar[st], (t / C::kStages) & 1)) {
      set_status(a.status, LG_ERR_TIMEOUT);
      ok = false;
      break;
    }
    const unsigned char *ks = smem + (size_t)st * 2 * C::kTileBytes;
    const unsigned char *vs = ks + C::kTileBytes;
#pragma unroll
    for (int step = 0; step < C::kSteps; ++step) {
      const int r = warp * C::kRowsPerWarp + step * C::kRPW + lane / LPR;  // row in tile
      const int rc = t * C::kTile + r;                                       // row in chunk
      const bool valid = rc < rows;
      const uint4 ku = *reinterpret_cast<const uint4 *>(ks + r * C::kRowBytes + li * 16);
      const uint4 vu = *reinterpret_cast<const uint4 *>(vs + r * C::kRowBytes + li * 16);
      float2 k2[NP], v2[NP];
      Elem<T>::unpack(ku, k2);
      Elem<T>::unpack(vu, v2);
      float part[GP];
#pragma unroll
      for (int g = 0; g < GP; ++g) {
        if (g < G) {
          float2 acc = make_float2(0.f, 0.f);
#pragma unroll
          for (int j = 0; j < NP; ++j) acc = ffma2(q2[g][j], k2[j], acc);
          part[g] = acc.x + acc.y;
        } else {
          part[g] = 0.f;
        }
      }
      HeadReduce<GP, LPR / 2>::run(part, lane);
      const float s = part[0];  // logit of head hd for this row, log2 units
      const bool live = valid && own;
      const bool need = live && s > m_ref;
      if (__any_sync(0xffffffffu, need)) {
        const float m_new = need ? s : m_ref;
        const float corr = m_new == m_ref ? 1.f : exp2f(m_ref - m_new);  // -inf -> 0
        u_acc = l_acc > 0.f ? corr * (u_acc + (m_ref - m_new) * l_acc) : 0.f;
        l_acc *= corr;
        sig *= corr;
        m_ref = m_new;
#pragma unroll
        for (int g = 0; g < G; ++g) {
          const float cg = __shfl_sync(0xffffffffu, corr, gbase + g * DUP);
          const float2 c2 = make_float2(cg, cg);
#pragma unroll
          for (int j = 0; j < NP; ++j) o2[g][j] = __fmul2_rn(o2[g][j], c2);
        }
      }
      // rows past the chunk end hold stale shared memory: they must not touch the sums
      const float p = live ? exp2f(s - m_ref) : 0.f;
      if (live) {
        l_acc += p;
        u_acc += p * (s - m_ref);
        if (row0 + rc >= suffix_lo) sig += p;
      }
      if (logits && live && (li % DUP) == 0) logits[(lrow0 + rc) * G + hd] = s;
      if (!valid) {
#pragma unroll
        for (int j = 0; j < NP; ++j) v2[j] = make_float2(0.f, 0.f);
      }
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const float pg = __shfl_sync(0xffffffffu, p, gbase + g * DUP);
        const float2 p2 = make_float2(pg, pg);
#pragma unroll
        for (int j = 0; j < NP; ++j) o2[g][j] = ffma2(p2, v2[j], o2[g][j]);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty_bar[st]);
  }

  // ---------------------------------------------------------------- CTA merge of row groups
  // all copies have landed (every tile was waited on), so the ring is free for scratch
  asm volatile("bar.sync 1, %0;" ::"n"(C::kWarps * 32) : "memory");
  if (!ok) return;
  float *so = reinterpret_cast<float *>(smem);            // [kGroups][G][D]
  float *ss = so + C::kGroups * G * D;                    // [kGroups][GP][4]
#pragma unroll
  for (int g = 0; g < G; ++g)
#pragma unroll
    for (int j = 0; j < NP; ++j) {
      float *dst = so + ((size_t)rgrp * G + g) * D + li * EPL + 2 * j;
      dst[0] = o2[g][j].x;
      dst[1] = o2[g][j].y;
    }
  if ((li % DUP) == 0) {
    float *dst = ss + ((size_t)rgrp * GP + hd) * 4;
    dst[0] = m_ref;
    dst[1] = l_acc;
    dst[2] = u_acc;
    dst[3] = sig;
  }
  asm volatile("bar.sync 1, %0;" ::"n"(C::kWarps * 32) : "memory");

  const int tid = threadIdx.x;
  const int64_t pbase = (((int64_t)lloc * a.batch + b) * a.H_q + (int64_t)kvh * G);
  for (int idx = tid; idx < G * D; idx += C::kWarps * 32) {
    const int g = idx / D, e = idx % D;
    float M = -INFINITY;
    for (int r = 0; r < C::kGroups; ++r) M = fmaxf(M, ss[(r * GP + g) * 4]);
    float o = 0.f, l = 0.f, u = 0.f, sg = 0.f;
    for (int r = 0; r < C::kGroups; ++r) {
      const float *st = ss + (r * GP + g) * 4;
      if (!(st[1] > 0.f)) continue;  // row group saw no row of this chunk
      const float f = exp2f(st[0] - M);
      o += f * so[((size_t)r * G + g) * D + e];
      if (e == 0) {
        l += f * st[1];
        u += f * (st[2] + (st[0] - M) * st[1]);
        sg += f * st[3];
      }
    }
    float *pp = a.partial + ((pbase + g) * a.max_chunks + chunk) * (D + 8);
    pp[8 + e] = o;
    if (e == 0) {
      pp[0] = M;
      pp[1] = l;
      pp[2] = u;
      pp[3] = sg;
    }
  }
}

// Merge the chunk partials of one (layer, sequence, query head): out = O / l and the
// statistics {m, l, H, S} in natural units.  One warp per head, eight heads per block.
template <typename T, int D>
__global__ void attend_combine_kernel(AttendArgs a, void *out, float *stats, float *final_ml) {
  pdl_enter();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t head = (int64_t)blockIdx.x * (blockDim.x >> 5) + warp;
  if (head >= (int64_t)a.n_layers * a.batch * a.H_q) return;
  if (status_bad(a.status)) return;
  const int b = (int)((head / a.H_q) % a.batch);
  const int n = a.len[b];
  if (n > a.max_len) return;
  constexpr int EPL = D / 32;
  if (n <= 0) {  // empty sequence: no attention; zero output, m = -inf
#pragma unroll
    for (int k = 0; k < EPL; ++k) Elem<T>::store(out, head * D + lane + 32 * k, 0.f);
    if (lane == 0) {
      stats[head * 4] = -INFINITY;
      stats[head * 4 + 1] = stats[head * 4 + 2] = stats[head * 4 + 3] = 0.f;
    }
    return;
  }
  const int nch = (n + a.chunk_rows - 1) / a.chunk_rows;
  const float *pp = a.partial + head * a.max_chunks * (D + 8);
  float M = -INFINITY;
  for (int j = 0; j < nch; ++j) M = fmaxf(M, pp[j * (D + 8)]);
  float l = 0.f, u = 0.f, sg = 0.f, o[EPL];
#pragma unroll
  for (int k = 0; k < EPL; ++k) o[k] = 0.f;
  for (int j = 0; j < nch; ++j) {
    const float *q = pp + j * (D + 8);
    const float f = exp2f(q[0] - M);
    l += f * q[1];
    u += f * (q[2] + (q[0] - M) * q[1]);
    sg += f * q[3];
#pragma unroll
    for (int k = 0; k < EPL; ++k) o[k] += f * q[8 + lane + 32 * k];
  }
  const float inv_l = 1.f / l;
#pragma unroll
  for (int k = 0; k < EPL; ++k) Elem<T>::store(out, head * D + lane + 32 * k, o[k] * inv_l);
  if (lane == 0) {
    constexpr float kLn2 = 0.69314718055994530942f;
    float *st = stats + head * 4;
    st[0] = M * kLn2;
    st[1] = l;
    st[2] = logf(l) - u * kLn2 * inv_l;
    st[3] = sg * inv_l;
    if (final_ml) {
      final_ml[head * 2] = M;
      final_ml[head * 2 + 1] = l;
    }
  }
}

constexpr int kH2ORows = 4;  // rows of the score update a thread has in flight

// H2O score: h2o[layer][kvh][slot] += sum over the heads of the group of a_i, from the logits
// kept by the partial pass and the merged (M, l) of every head.
template <int G>
__global__ void __launch_bounds__(256) h2o_accumulate_kernel(AttendArgs a, float *h2o,
                                                              const float *final_ml) {
  pdl_enter();
  const int kvh = blockIdx.y, b = blockIdx.z % a.batch, lloc = blockIdx.z / a.batch;
  const int layer = a.layer0 + lloc;
  if (status_bad(a.status)) return;
  const int n = a.len[b];
  if (n > a.max_len) return;
  float M[G], inv_l[G];
  const int64_t head0 = ((int64_t)lloc * a.batch + b) * a.H_q + (int64_t)kvh * G;
#pragma unroll
  for (int g = 0; g < G; ++g) {
    M[g] = final_ml[(head0 + g) * 2];
    inv_l[g] = 1.f / final_ml[(head0 + g) * 2 + 1];
  }
  const int64_t lrow0 = ((int64_t)lloc * a.H_kv + kvh) * a.S_total + a.seq_off[b];
  float *sc = h2o + ((int64_t)layer * a.H_kv + kvh) * a.S_total + a.seq_off[b];
  // kH2ORows rows per thread with all their loads in flight; a row's G logits in 16- or 8-byte
  // loads where G allows (the logits start 256-byte aligned, a row at a multiple of 4 G bytes)
  const int stride = gridDim.x * blockDim.x;
  for (int i0 = blockIdx.x * blockDim.x + threadIdx.x; i0 < n; i0 += kH2ORows * stride) {
    float lg[kH2ORows][G], old[kH2ORows];
#pragma unroll
    for (int k = 0; k < kH2ORows; ++k) {
      const int i = i0 + k * stride;
      if (i < n) {
        const float *src = a.logits + (lrow0 + i) * G;
        if (G % 4 == 0) {
#pragma unroll
          for (int g = 0; g < G; g += 4) {
            const float4 v = *reinterpret_cast<const float4 *>(src + g);
            lg[k][g] = v.x, lg[k][g + 1] = v.y, lg[k][g + 2] = v.z, lg[k][g + 3] = v.w;
          }
        } else if (G % 2 == 0) {
#pragma unroll
          for (int g = 0; g < G; g += 2) {
            const float2 v = *reinterpret_cast<const float2 *>(src + g);
            lg[k][g] = v.x, lg[k][g + 1] = v.y;
          }
        } else {
#pragma unroll
          for (int g = 0; g < G; ++g) lg[k][g] = src[g];
        }
        old[k] = sc[i];
      }
    }
#pragma unroll
    for (int k = 0; k < kH2ORows; ++k) {
      const int i = i0 + k * stride;
      if (i < n) {
        float acc = 0.f;
#pragma unroll
        for (int g = 0; g < G; ++g) acc += exp2f(lg[k][g] - M[g]) * inv_l[g];
        sc[i] = old[k] + acc;
      }
    }
  }
}

// ------------------------------------------------------------------ launch

template <typename T, int D, int G>
static cudaError_t launch_typed(const AttendArgs &a, int64_t rows_total, void *out, float *stats,
                                float *final_ml, float *h2o, cudaStream_t s) {
  using C = AttendCfg<T, D, G>;
  cudaError_t e;
  if (Elem<T>::kDtype == LG_BF16) {
    // tensor-core partial pass (lg_attend_mma.cu)
    e = launch_attend_mma_partial(a, D, G, rows_total, s);
    if (e != cudaSuccess) return e;
  } else {
    auto kp = attend_partial_kernel<T, D, G>;
    e = cudaFuncSetAttribute(kp, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
    if (e != cudaSuccess) return e;
    dim3 grid(a.max_chunks, a.H_kv, a.n_layers * a.batch);
    LG_TRY(launch_pdl(kp, grid, C::kThreads, C::kSmem, s, a));
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (Elem<T>::kDtype != LG_BF16) {
    // the tensor-core pass merges its chunk partials itself
    const int64_t heads = (int64_t)a.n_layers * a.batch * a.H_q;
    LG_TRY(launch_pdl(attend_combine_kernel<T, D>, (unsigned)((heads + 7) / 8), 256, 0, s, a, out,
                      stats, final_ml));
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (h2o) {
    // at most 16 CTAs a (layer, sequence, kv-head) stream: up to 16 K rows a stream leave each
    // thread its kH2ORows rows in flight (a grid sized for one row a thread ran with half the
    // warps resident and most of its CTAs idle on short sequences)
    int gx = (a.max_len + 256 * kH2ORows - 1) / (256 * kH2ORows);
    if (gx > 16) gx = 16;
    LG_TRY(launch_pdl(h2o_accumulate_kernel<G>, dim3(gx, a.H_kv, a.n_layers * a.batch), 256, 0, s,
                      a, h2o, final_ml));
    e = cudaGetLastError();
  }
  return e;
}

template <typename T, int D>
static cudaError_t launch_d(const AttendArgs &a, int64_t rt, int g, void *out, float *stats,
                            float *fm, float *h2o, cudaStream_t s) {
  switch (g) {
    case 1: return launch_typed<T, D, 1>(a, rt, out, stats, fm, h2o, s);
    case 2: return launch_typed<T, D, 2>(a, rt, out, stats, fm, h2o, s);
    case 3: return launch_typed<T, D, 3>(a, rt, out, stats, fm, h2o, s);
    case 4: return launch_typed<T, D, 4>(a, rt, out, stats, fm, h2o, s);
    case 5: return launch_typed<T, D, 5>(a, rt, out, stats, fm, h2o, s);
    case 6: return launch_typed<T, D, 6>(a, rt, out, stats, fm, h2o, s);
    case 7: return launch_typed<T, D, 7>(a, rt, out, stats, fm, h2o, s);
    case 8: return launch_typed<T, D, 8>(a, rt, out, stats, fm, h2o, s);
  }
  return cudaErrorInvalidValue;
}

// rows per staging tile: the tensor-core path streams 128-row tiles; the fp32 path 8 KB tiles
int attend_tile_rows(int dtype, int d) {
  if (dtype == LG_BF16) return mma_tile_rows();
  return 8192 / (d * 4);
}

cudaError_t launch_attend(const AttendArgs &a, int dtype, int d, int g, int64_t rows_total,
                          void *out, float *stats, float *final_ml, float *h2o, cudaStream_t s) {
  if (dtype == LG_BF16 && d == 128)
    return launch_d<__nv_bfloat16, 128>(a, rows_total, g, out, stats, final_ml, h2o, s);
  if (dtype == LG_BF16 && d == 64)
    return launch_d<__nv_bfloat16, 64>(a, rows_total, g, out, stats, final_ml, h2o, s);
  if (dtype == LG_F32 && d == 128)
    return launch_d<float, 128>(a, rows_total, g, out, stats, final_ml, h2o, s);
  if (dtype == LG_F32 && d == 64)
    return launch_d<float, 64>(a, rows_total, g, out, stats, final_ml, h2o, s);
  return cudaErrorInvalidValue;
}

}  // namespace lg
