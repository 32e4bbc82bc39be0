// Device side of the synthetic workload generator (harness).  Same recipe and
// same source of truth as the host side: synth_core.h.  Build with
// --fmad=false so that no multiply-add is fused.
#include <cuda_runtime.h>

#include "synth_core.h"

namespace {

// The per-step harness kernels (selection of each sequence's inputs, advance) sit between the
// guard's kernels, which are launched with programmatic stream serialization; they are launched
// the same way and wait (griddepcontrol.wait) for the kernel before them before touching memory.
__device__ __forceinline__ void pdl_enter() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, cudaStream_t s,
                       Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

__device__ __forceinline__ void store(const syn_workload &w, void *out, int64_t i, float v) {
  if (w.dtype == SYN_BF16)
    ((uint16_t *)out)[i] = syn_bf16_bits(v);
  else
    ((float *)out)[i] = v;
}

// grid: x = row block, y = layer * H_kv + kvh, z = sequence; one thread per element
__global__ void fill_cache_kernel(syn_workload w, const syn_seq *seqs, const int64_t *seq_off,
                                  const int32_t *n_rows, int64_t S_total, void *K, void *V) {
  const int b = blockIdx.z, lh = blockIdx.y;
  const int layer = lh / w.H_kv, kvh = lh % w.H_kv;
  const int rows_per_block = blockDim.x / w.d;
  const int r = threadIdx.x / w.d, e = threadIdx.x % w.d;
  const syn_seq s = seqs[b];
  const int64_t nr = n_rows[b];
  for (int64_t p = (int64_t)blockIdx.x * rows_per_block + r; p < nr;
       p += (int64_t)gridDim.x * rows_per_block) {
    int64_t i = ((int64_t)lh * S_total + seq_off[b] + p) * w.d + e;
    store(w, K, i, syn_row_value(&w, &s, 0, layer, kvh, b, p, e));
    store(w, V, i, syn_row_value(&w, &s, 1, layer, kvh, b, p, e));
  }
}

// one thread per (layer, sequence, query head) for q, per (layer, sequence, kv-head, element)
// for the new K/V rows.  mode 0: as the sequence state says; 1: every sequence loop-free;
// 2: as if no sequence had been intervened on.
__global__ void step_q_kernel(syn_workload w, const syn_seq *seqs, int batch, const int64_t *pos,
                              int mode, void *q) {
  int t = blockIdx.x * blockDim.x + threadIdx.x;
  int total = w.L * batch * w.H_q;
  if (t >= total) return;
  int h = t % w.H_q, b = (t / w.H_q) % batch, layer = t / (w.H_q * batch);
  syn_seq s = seqs[b];
  if (mode == 1) s.fresh_from = 0;
  if (mode == 2) s.fresh_from = SYN_NEVER;
  float qv[128];
  syn_query(&w, &s, layer, h, b, pos[b], qv);
  for (int e = 0; e < w.d; ++e) store(w, q, (int64_t)t * w.d + e, qv[e]);
}

__global__ void step_kv_kernel(syn_workload w, const syn_seq *seqs, int batch,
                               const int64_t *pos, int mode, void *k_new, void *v_new) {
  int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  int64_t total = (int64_t)w.L * batch * w.H_kv * w.d;
  if (t >= total) return;
  int e = t % w.d;
  int kvh = (t / w.d) % w.H_kv;
  int b = (t / ((int64_t)w.d * w.H_kv)) % batch;
  int layer = t / ((int64_t)w.d * w.H_kv * batch);
  syn_seq s = seqs[b];
  if (mode == 1) s.fresh_from = 0;
  if (mode == 2) s.fresh_from = SYN_NEVER;
  store(w, k_new, t, syn_row_value(&w, &s, 0, layer, kvh, b, pos[b], e));
  store(w, v_new, t, syn_row_value(&w, &s, 1, layer, kvh, b, pos[b], e));
}

// the three selections of one step (q, k_new, v_new) in one launch
struct Sel3 {
  const char *loop[3];
  const char *fresh[3];
  char *out[3];
  int64_t chunks[3];  // 16-byte chunks per (layer, sequence) row of each tensor
  // nullable: each sequence's token id and top-1 probability of the step, both variants
  const int32_t *tok_loop, *tok_fresh;
  const float *pm_loop, *pm_fresh;
  int32_t *tok;
  float *pm;
};

// Whether sequence b takes the loop-free variant this step: once the guard has intervened on
// it (the guard state's intervention count, word n_int_word of its state_words-word record, is
// positive), its next tokens are loop-free; without a guard state (the comparator policies)
// loops persist.
__device__ __forceinline__ bool fresh_variant(const int32_t *state, int state_words, int n_int_word,
                                              int b) {
  return state && state[(int64_t)b * state_words + n_int_word] > 0;
}

__global__ void select3_kernel(const int32_t *state, int state_words, int n_int_word, int batch,
                               int L, Sel3 s) {
  pdl_enter();
  int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (s.tok && t < batch) {
    const int b = (int)t;
    const bool fresh = fresh_variant(state, state_words, n_int_word, b);
    s.tok[b] = fresh ? s.tok_fresh[b] : s.tok_loop[b];
    s.pm[b] = fresh ? s.pm_fresh[b] : s.pm_loop[b];
  }
  for (int k = 0; k < 3; ++k) {
    const int64_t total = (int64_t)L * batch * s.chunks[k];
    if (t < total) {
      const int b = (int)((t / s.chunks[k]) % batch);
      const char *src = fresh_variant(state, state_words, n_int_word, b) ? s.fresh[k] : s.loop[k];
      ((uint4 *)s.out[k])[t] = ((const uint4 *)src)[t];
      return;
    }
    t -= total;
  }
}

// Read-only streaming pass (harness, not part of the generator's recipe): every 16-byte word of
// the buffer is loaded once with an evict-first hint and folded by XOR into one word per warp,
// so the loads cannot be dropped.  bench.py times it as the read-only bandwidth denominator
// beside the copy peak (a decode pass reads its K/V and writes next to nothing).  Grid-stride,
// eight independent 16-byte loads in flight per thread.
__global__ void __launch_bounds__(256) read_stream_kernel(const uint4 *p, int64_t n16,
                                                          unsigned *sink) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  unsigned acc = 0;
  for (; i + 7 * stride < n16; i += 8 * stride) {
    uint4 v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = __ldcs(p + i + k * stride);
#pragma unroll
    for (int k = 0; k < 8; ++k) acc ^= v[k].x ^ v[k].y ^ v[k].z ^ v[k].w;
  }
  for (; i < n16; i += stride) {
    const uint4 v = __ldcs(p + i);
    acc ^= v.x ^ v.y ^ v.z ^ v.w;
  }
  acc = __reduce_xor_sync(0xffffffffu, acc);
  if ((threadIdx.x & 31) == 0) atomicXor(sink, acc);
}

// Read-only pass with 1-D bulk (TMA) copies: one warp per CTA streams blocks of `block` bytes
// (grid-stride) through a ring of 4 shared-memory stages, each copy completing on its stage's
// mbarrier; lane j folds word j of every block into its XOR.  Every wait is bounded (2 s of
// %globaltimer): on a timeout the CTA records it in *err, waits (bounded) for its copies in
// flight and returns.
constexpr int kReadStages = 4;

__device__ __forceinline__ uint32_t rd_smem(const void *p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ bool rd_try_wait(uint64_t *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(rd_smem(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool rd_wait(uint64_t *bar, uint32_t parity) {
  uint64_t t0, t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
  while (!rd_try_wait(bar, parity)) {
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    if (t - t0 > 2000000000ull) return false;
  }
  return true;
}

__device__ __forceinline__ void rd_issue(uint64_t *bar, void *dst, const void *src, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(rd_smem(bar)),
               "r"(bytes)
               : "memory");
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(rd_smem(dst)), "l"(src), "r"(bytes), "r"(rd_smem(bar))
      : "memory");
}

__global__ void __launch_bounds__(32) read_bulk_kernel(const unsigned char *p, int64_t nblocks,
                                                       int block, unsigned *sink, int *err) {
  extern __shared__ __align__(128) unsigned char rbuf[];
  __shared__ __align__(8) uint64_t bar[kReadStages];
  const int lane = threadIdx.x;
  if (lane == 0) {
    for (int k = 0; k < kReadStages; ++k)
      asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(rd_smem(&bar[k])) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  __syncwarp();
  const int64_t g = gridDim.x;
  if (lane == 0)
    for (int k = 0; k < kReadStages; ++k) {
      const int64_t blk = blockIdx.x + k * g;
      if (blk < nblocks) rd_issue(&bar[k], rbuf + k * block, p + blk * block, block);
    }
  unsigned acc = 0;
  int64_t i = 0;
  bool ok = true;
  for (;; ++i) {
    const int64_t blk = blockIdx.x + i * g;
    if (blk >= nblocks) break;
    const int k = (int)(i % kReadStages);
    const uint32_t parity = (uint32_t)((i / kReadStages) & 1);
    ok = rd_wait(&bar[k], parity);
    if (!__all_sync(0xffffffffu, ok)) {
      ok = false;
      break;
    }
    acc ^= ((const unsigned *)(rbuf + k * block))[lane];
    __syncwarp();
    const int64_t nxt = blk + kReadStages * g;
    if (lane == 0 && nxt < nblocks) rd_issue(&bar[k], rbuf + k * block, p + nxt * block, block);
  }
  if (!ok) {
    if (lane == 0) atomicExch(err, 1);
    // the copies still in flight: blocks i .. i + kReadStages - 1 (those that exist)
    for (int64_t j = i; j < i + kReadStages; ++j) {
      const int64_t blk = blockIdx.x + j * g;
      if (blk >= nblocks) break;
      rd_wait(&bar[j % kReadStages], (uint32_t)((j / kReadStages) & 1));
    }
    return;
  }
  acc = __reduce_xor_sync(0xffffffffu, acc);
  if (lane == 0) atomicXor(sink, acc);
}
}  // namespace

extern "C" {

int syn_dev_select3(const int32_t *state, int state_words, int n_int_word, int batch, int L,
                    const int64_t *rowlen_bytes, const void *const *loop_bufs,
                    const void *const *fresh_bufs, void *const *outs, const int32_t *tok_loop,
                    const int32_t *tok_fresh, const float *pm_loop, const float *pm_fresh,
                    int32_t *tok, float *pm, cudaStream_t stream) {
  Sel3 s;
  if (tok && (!tok_loop || !tok_fresh || !pm_loop || !pm_fresh || !pm)) return 1;
  s.tok_loop = tok_loop;
  s.tok_fresh = tok_fresh;
  s.pm_loop = pm_loop;
  s.pm_fresh = pm_fresh;
  s.tok = tok;
  s.pm = pm;
  int64_t total = 0;
  for (int k = 0; k < 3; ++k) {
    if (rowlen_bytes[k] % 16) return 1;
    s.loop[k] = (const char *)loop_bufs[k];
    s.fresh[k] = (const char *)fresh_bufs[k];
    s.out[k] = (char *)outs[k];
    s.chunks[k] = rowlen_bytes[k] / 16;
    total += (int64_t)L * batch * s.chunks[k];
  }
  return launch_pdl(select3_kernel, dim3((unsigned)((total + 255) / 256)), dim3(256), stream,
                    state, state_words, n_int_word, batch, L, s) == cudaSuccess
             ? 0
             : 2;
}

int syn_dev_fill_cache(const syn_workload *w, const syn_seq *seqs_dev, int batch,
                       const int64_t *seq_off_dev, const int32_t *n_rows_dev, int64_t S_total,
                       int max_rows, void *K, void *V, cudaStream_t stream) {
  if (w->d > 128 || 256 % w->d) return 1;
  int rows_per_block = 256 / w->d;
  int gx = (max_rows + rows_per_block - 1) / rows_per_block;
  if (gx > 4096) gx = 4096;
  if (gx < 1) gx = 1;
  dim3 grid(gx, w->L * w->H_kv, batch);
  fill_cache_kernel<<<grid, 256, 0, stream>>>(*w, seqs_dev, seq_off_dev, n_rows_dev, S_total, K, V);
  return cudaGetLastError() == cudaSuccess ? 0 : 2;
}

int syn_dev_step(const syn_workload *w, const syn_seq *seqs_dev, int batch, const int64_t *pos_dev,
                 int mode, void *q, void *k_new, void *v_new, cudaStream_t stream) {
  if (w->d > 128) return 1;
  int nq = w->L * batch * w->H_q;
  step_q_kernel<<<(nq + 127) / 128, 128, 0, stream>>>(*w, seqs_dev, batch, pos_dev, mode, q);
  int64_t nkv = (int64_t)w->L * batch * w->H_kv * w->d;
  step_kv_kernel<<<(unsigned)((nkv + 255) / 256), 256, 0, stream>>>(*w, seqs_dev, batch, pos_dev,
                                                                    mode, k_new, v_new);
  return cudaGetLastError() == cudaSuccess ? 0 : 2;
}

// one read-only pass over bytes (a multiple of 16, 16-byte aligned) of device memory; ctas = the
// grid (a multiple of the SM count); sink: one device word, XOR of everything read
int syn_dev_read_stream(const void *p, int64_t bytes, unsigned *sink, int ctas,
                        cudaStream_t stream) {
  if (!p || !sink || bytes % 16 || ((uintptr_t)p & 15) || ctas < 1) return 1;
  read_stream_kernel<<<ctas, 256, 0, stream>>>((const uint4 *)p, bytes / 16, sink);
  return cudaGetLastError() == cudaSuccess ? 0 : 2;
}

// the same pass with 1-D bulk copies into shared memory: block bytes per copy (a multiple of
// 16, at most 32768), bytes a multiple of block; err: one device word, set on a timed-out wait
int syn_dev_read_bulk(const void *p, int64_t bytes, int block, unsigned *sink, int *err,
                      int ctas, cudaStream_t stream) {
  if (!p || !sink || !err || block < 128 || block > 32768 || block % 16 || bytes % block ||
      ((uintptr_t)p & 15) || ctas < 1)
    return 1;
  const int smem = kReadStages * block;
  if (cudaFuncSetAttribute(read_bulk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) !=
      cudaSuccess)
    return 2;
  read_bulk_kernel<<<ctas, 32, smem, stream>>>((const unsigned char *)p, bytes / block, block,
                                               sink, err);
  return cudaGetLastError() == cudaSuccess ? 0 : 2;
}

}  // extern "C"
