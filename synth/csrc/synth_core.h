/*
 * synth_core.h -- counter-based synthetic workload generator.
 *
 * This is harness code shared by the host generator (synth_host.cpp, built
 * with g++ -ffp-contract=off) and the device generator (synth_dev.cu, built
 * with nvcc --fmad=false).  Both compile exactly these functions, so a value
 * drawn on the host and on the GPU has the same bits.  It holds none of the
 * guard's arithmetic: only hashing, Irwin-Hall normals, loop planting and the
 * rounding of values to the cache dtype.
 *
 * Recipe (every float op is a single IEEE round-to-nearest op, no FMA):
 *   mix(x)        splitmix64 finaliser (Steele, Lea, Flood 2014)
 *   key           mix(mix(seed) ^ id(role, layer, head, seq))
 *   normal(k, i)  h0 = mix(k ^ 2i), h1 = mix(k ^ (2i+1)); four 24-bit fields
 *                 summed as integers S; z = float(S - 2^25) * sqrt(3)/2^24,
 *                 i.e. Irwin-Hall(4) rescaled to unit variance.
 *   base row      scale(layer, kv-head) * z, keys of the first n_sink
 *                 positions multiplied by sink_factor
 *   loop row      base(src) + sigma * z', src = start - P + ((p - start) mod P)
 *   query         token p inside the loop: k~ = stored key at src(p), the key p repeats;
 *                   zstar mode: q = (zstar*sqrt(d) / |k~|^2) k~ + q_noise z
 *                   literal mode: q = k~ + q_noise z
 *                 otherwise q = z
 */
#pragma once
#include <math.h>
#include <stdint.h>

#ifdef __CUDACC__
#define SYN_HD __host__ __device__ __forceinline__
#else
#define SYN_HD static inline
#endif

enum {
  SYN_ROLE_K = 1,       /* base key rows             */
  SYN_ROLE_V = 2,       /* base value rows           */
  SYN_ROLE_NK = 3,      /* loop noise on keys        */
  SYN_ROLE_NV = 4,      /* loop noise on values      */
  SYN_ROLE_Q = 5,       /* query noise / fresh query */
  SYN_ROLE_SCALE_K = 6, /* per-(layer, kv-head) key scale   */
  SYN_ROLE_SCALE_V = 7  /* per-(layer, kv-head) value scale */
};

enum { SYN_BF16 = 0, SYN_F32 = 1 };
enum { SYN_Q_ZSTAR = 0, SYN_Q_LITERAL = 1 };

#define SYN_NEVER 0x7fffffff

typedef struct {
  uint64_t seed;
  int32_t L, H_q, H_kv, d, dtype;
  int32_t head_scale;  /* 1: scale ~ U(0.5, 2) per (layer, kv-head); 0: 1.0 */
  int32_t n_sink;      /* keys at positions < n_sink are multiplied by sink_factor */
  float sink_factor;
  float sigma;         /* loop noise standard deviation */
  int32_t query_mode;  /* SYN_Q_ZSTAR or SYN_Q_LITERAL */
  float zstar;         /* target logit of every loop copy (zstar mode) */
  float q_noise;       /* query noise standard deviation */
  int32_t pad;
} syn_workload;

typedef struct {
  int32_t looping;     /* 1: rows at positions >= start repeat with period P */
  int32_t start;       /* first looping position */
  int32_t period;      /* P */
  int32_t fresh_from;  /* rows/queries at positions >= fresh_from are loop-free */
} syn_seq;

SYN_HD uint64_t syn_mix(uint64_t x) {
  x += 0x9E3779B97F4A7C15ull;
  x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
  x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
  return x ^ (x >> 31);
}

SYN_HD uint64_t syn_key(uint64_t seed, int role, int layer, int head, int seq) {
  uint64_t id = (((uint64_t)role * 64u + (uint64_t)layer) * 256u + (uint64_t)head) * 65536u +
                (uint64_t)seq;
  return syn_mix(syn_mix(seed) ^ id);
}

SYN_HD float syn_u32_as_float(uint32_t u) {
#ifdef __CUDA_ARCH__
  return __uint_as_float(u);
#else
  union { uint32_t u; float f; } c;
  c.u = u;
  return c.f;
#endif
}

SYN_HD uint32_t syn_float_as_u32(float f) {
#ifdef __CUDA_ARCH__
  return __float_as_uint(f);
#else
  union { uint32_t u; float f; } c;
  c.f = f;
  return c.u;
#endif
}

/* sqrt(3) / 2^24 rounded to fp32 (bits 0x33ddb3d7) */
#define SYN_NORMAL_C_BITS 0x33ddb3d7u

SYN_HD float syn_normal(uint64_t key, uint64_t idx) {
  uint64_t h0 = syn_mix(key ^ (2u * idx));
  uint64_t h1 = syn_mix(key ^ (2u * idx + 1u));
  int64_t s = (int64_t)(h0 >> 40) + (int64_t)((h0 >> 16) & 0xFFFFFFu) + (int64_t)(h1 >> 40) +
              (int64_t)((h1 >> 16) & 0xFFFFFFu);
  float x = (float)(s - ((int64_t)1 << 25));
  return x * syn_u32_as_float(SYN_NORMAL_C_BITS);
}

/* uniform in [0, 1) with 24 bits, exact in fp32 */
SYN_HD float syn_uniform(uint64_t key, uint64_t idx) {
  uint64_t h = syn_mix(key ^ idx);
  return (float)(int32_t)(h >> 40) * syn_u32_as_float(0x33800000u); /* 2^-24 */
}

/* float -> bf16 bits, round to nearest even (inputs are finite) */
SYN_HD uint16_t syn_bf16_bits(float f) {
  uint32_t u = syn_float_as_u32(f);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

SYN_HD float syn_bf16_value(uint16_t b) { return syn_u32_as_float((uint32_t)b << 16); }

/* value as stored in the cache dtype, widened back to float */
SYN_HD float syn_stored(const syn_workload *w, float v) {
  return w->dtype == SYN_BF16 ? syn_bf16_value(syn_bf16_bits(v)) : v;
}

SYN_HD float syn_scale(const syn_workload *w, int is_value, int layer, int kvh) {
  if (!w->head_scale) return 1.0f;
  float u = syn_uniform(syn_key(w->seed, is_value ? SYN_ROLE_SCALE_V : SYN_ROLE_SCALE_K, layer,
                                kvh, 0),
                        0);
  return u * 1.5f + 0.5f;
}

/* base (non-loop) value of element e of the K (is_value=0) or V row at position p */
SYN_HD float syn_base(const syn_workload *w, int is_value, int layer, int kvh, int seq, int64_t p,
                      int e) {
  float z = syn_normal(syn_key(w->seed, is_value ? SYN_ROLE_V : SYN_ROLE_K, layer, kvh, seq),
                       (uint64_t)p * (uint64_t)w->d + (uint64_t)e);
  float v = z * syn_scale(w, is_value, layer, kvh);
  if (!is_value && p < w->n_sink) v = v * w->sink_factor;
  return v;
}

SYN_HD int syn_loop_active(const syn_seq *s, int64_t p) {
  return s->looping && p >= s->start && p < s->fresh_from;
}

SYN_HD int64_t syn_loop_src(const syn_seq *s, int64_t p) {
  return (int64_t)s->start - s->period + ((p - s->start) % s->period);
}

/* value (before rounding to the cache dtype) of element e of the row at position p */
SYN_HD float syn_row_value(const syn_workload *w, const syn_seq *s, int is_value, int layer,
                           int kvh, int seq, int64_t p, int e) {
  if (syn_loop_active(s, p)) {
    float v = syn_base(w, is_value, layer, kvh, seq, syn_loop_src(s, p), e);
    float n = syn_normal(syn_key(w->seed, is_value ? SYN_ROLE_NV : SYN_ROLE_NK, layer, kvh, seq),
                         (uint64_t)p * (uint64_t)w->d + (uint64_t)e);
    return v + n * w->sigma;
  }
  return syn_base(w, is_value, layer, kvh, seq, p, e);
}

/* query of head h for the token at position p (the one appended this step); q[d] is the value
   before rounding to the cache dtype. */
SYN_HD void syn_query(const syn_workload *w, const syn_seq *s, int layer, int h, int seq,
                      int64_t p, float *q) {
  int g = w->H_q / w->H_kv;
  int kvh = h / g;
  uint64_t qk = syn_key(w->seed, SYN_ROLE_Q, layer, h, seq);
  /* the token at p is a loop row: its query targets the key it repeats, k~ = base(src(p)) */
  if (syn_loop_active(s, p)) {
    int64_t src = syn_loop_src(s, p);
    if (w->query_mode == SYN_Q_LITERAL) {
      for (int e = 0; e < w->d; ++e) {
        float kt = syn_stored(w, syn_base(w, 0, layer, kvh, seq, src, e));
        float z = syn_normal(qk, (uint64_t)p * (uint64_t)w->d + (uint64_t)e);
        q[e] = kt + z * w->q_noise;
      }
    } else {
      float nrm = 0.0f;
      for (int e = 0; e < w->d; ++e) {
        float kt = syn_stored(w, syn_base(w, 0, layer, kvh, seq, src, e));
        nrm = nrm + kt * kt;
      }
      float coef = (w->zstar * sqrtf((float)w->d)) / nrm;
      for (int e = 0; e < w->d; ++e) {
        float kt = syn_stored(w, syn_base(w, 0, layer, kvh, seq, src, e));
        float z = syn_normal(qk, (uint64_t)p * (uint64_t)w->d + (uint64_t)e);
        q[e] = coef * kt + z * w->q_noise;
      }
    }
  } else {
    for (int e = 0; e < w->d; ++e) q[e] = syn_normal(qk, (uint64_t)p * (uint64_t)w->d + (uint64_t)e);
  }
}
