/*
 * Seeded synthetic inputs for the routed-expert step of one MoE decoder layer.
 *
 * This file only generates inputs: expert payloads as canonical GGUF Q8_0 / Q4_0
 * block bytes, router weights, activations and route sets.  It holds none of the
 * step's arithmetic (no dequantisation, no dot product, no routing decision, no
 * cache logic).  Both the CPU oracle and the CUDA path are fed from it.
 *
 * Randomness is counter based: value number c of the stream named by a 64-bit key
 * is the SplitMix64 output function (Steele, Lea & Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014) applied to key + (c+1)*gamma, with
 * gamma = 0x9E3779B97F4A7C15.  Any (layer, expert, tensor, block) can therefore be
 * regenerated without storing the whole pack.
 *
 * Block layouts (GGUF, the format the paper serves, Background section):
 *   Q8_0: { fp16 d; int8 q[32]; }            34 bytes, weight = d * q
 *   Q4_0: { fp16 d; uint8 qs[16]; }          18 bytes, byte j holds element j in its
 *                                            low nibble and element j+16 in its high one
 * An expert payload is gate [I rows x H cols], up [I x H], down [H x I], each tensor
 * row-major with its 32-element blocks running along the column (input) dimension.
 *
 * Distributions (the workload recipe): quants uniform integers in [-127,127] (Q8_0)
 * or [0,15] (Q4_0 nibbles); scale d = RNE_fp16(|0.02 * N(0,1)|), subnormals kept.
 * Compile with -ffp-contract=off so x86-64 and aarch64 give the same bytes.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#define SYN_Q8_0 8
#define SYN_Q4_0 2

static const uint64_t GAMMA = 0x9E3779B97F4A7C15ULL;

static inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

/* value number ctr of stream key */
static inline uint64_t draw(uint64_t key, uint64_t ctr) { return mix64(key + (ctr + 1) * GAMMA); }

uint64_t syn_key(uint64_t seed, uint64_t domain, uint64_t a, uint64_t b, uint64_t c) {
  uint64_t k = mix64(seed + GAMMA);
  k = mix64(k ^ (domain + 1) * GAMMA);
  k = mix64(k ^ (a + 1) * GAMMA);
  k = mix64(k ^ (b + 1) * GAMMA);
  k = mix64(k ^ (c + 1) * GAMMA);
  return k;
}

uint64_t syn_draw(uint64_t key, uint64_t ctr) { return draw(key, ctr); }

/* uniform in [0,1) with 53 random bits */
static inline double unif(uint64_t r) { return (double)(r >> 11) * 0x1.0p-53; }

/* standard normal from two counter values (Box-Muller, first output) */
static inline double normal2(uint64_t key, uint64_t ctr) {
  double u1 = ((double)(draw(key, ctr) >> 11) + 1.0) * 0x1.0p-53; /* (0,1] */
  double u2 = unif(draw(key, ctr + 1));
  return sqrt(-2.0 * log(u1)) * cos(6.283185307179586 * u2);
}

/* double -> IEEE binary16, round to nearest even, subnormals kept; |v| < 65520 */
uint16_t syn_f64_to_f16(double v) {
  uint16_t sign = (v < 0 || (v == 0 && signbit(v))) ? 0x8000 : 0;
  double a = fabs(v);
  if (a == 0.0) return sign;
  if (a >= 65520.0) return sign | 0x7C00; /* rounds to infinity */
  int e;
  (void)frexp(a, &e); /* a in [2^(e-1), 2^e) */
  int eu = e - 1;
  if (eu < -14) { /* subnormal range: unit 2^-24 */
    double r = nearbyint(ldexp(a, 24));
    return sign | (uint16_t)r; /* r == 1024 encodes the smallest normal */
  }
  double r = nearbyint(ldexp(a, 10 - eu)); /* in [1024, 2048] */
  return sign | (uint16_t)(((eu + 15) << 10) + ((int)r - 1024));
}

uint64_t syn_block_bytes(int qtype) { return qtype == SYN_Q8_0 ? 34 : (qtype == SYN_Q4_0 ? 18 : 0); }

uint64_t syn_tensor_bytes(int rows, int cols, int qtype) {
  return (uint64_t)rows * (uint64_t)(cols / 32) * syn_block_bytes(qtype);
}

uint64_t syn_payload_bytes(int hidden, int inter, int qtype) {
  return 2 * syn_tensor_bytes(inter, hidden, qtype) + syn_tensor_bytes(hidden, inter, qtype);
}

/* One quantised tensor [rows x cols] of expert (layer, expert), tensor 0=gate 1=up 2=down. */
int syn_q_tensor(uint64_t seed, int layer, int expert, int tensor, int rows, int cols, int qtype,
                 uint8_t* out) {
  if (cols % 32 != 0 || rows <= 0 || (qtype != SYN_Q8_0 && qtype != SYN_Q4_0)) return -1;
  const uint64_t key = syn_key(seed, 1, (uint64_t)layer, (uint64_t)expert, (uint64_t)tensor);
  const int64_t nb = (int64_t)rows * (cols / 32);
  const uint64_t bb = syn_block_bytes(qtype);
#pragma omp parallel for schedule(static)
  for (int64_t b = 0; b < nb; ++b) {
    uint8_t* blk = out + (uint64_t)b * bb;
    const uint64_t c0 = (uint64_t)b * 20;
    uint16_t d = syn_f64_to_f16(fabs(0.02 * normal2(key, c0)));
    blk[0] = (uint8_t)(d & 0xFF);
    blk[1] = (uint8_t)(d >> 8);
    if (qtype == SYN_Q8_0) {
      for (int i = 0; i < 16; ++i) {
        uint64_t r = draw(key, c0 + 2 + i);
        uint32_t lo = (uint32_t)r, hi = (uint32_t)(r >> 32);
        int q0 = (int)(((uint64_t)lo * 255u) >> 32) - 127;
        int q1 = (int)(((uint64_t)hi * 255u) >> 32) - 127;
        blk[2 + 2 * i] = (uint8_t)(int8_t)q0;
        blk[3 + 2 * i] = (uint8_t)(int8_t)q1;
      }
    } else {
      uint64_t r0 = draw(key, c0 + 2), r1 = draw(key, c0 + 3);
      for (int i = 0; i < 8; ++i) {
        blk[2 + i] = (uint8_t)(r0 >> (8 * i));
        blk[10 + i] = (uint8_t)(r1 >> (8 * i));
      }
    }
  }
  return 0;
}

/* Whole expert payload: gate [I x H], up [I x H], down [H x I] back to back. */
int syn_payload(uint64_t seed, int layer, int expert, int hidden, int inter, int qtype, uint8_t* out) {
  uint64_t tb = syn_tensor_bytes(inter, hidden, qtype);
  if (syn_q_tensor(seed, layer, expert, 0, inter, hidden, qtype, out)) return -1;
  if (syn_q_tensor(seed, layer, expert, 1, inter, hidden, qtype, out + tb)) return -1;
  if (syn_q_tensor(seed, layer, expert, 2, hidden, inter, qtype, out + 2 * tb)) return -1;
  return 0;
}

/* out[i] = (float)(scale * N(0,1)), i < n, from stream key */
void syn_normal_f32(uint64_t key, double scale, int64_t n, float* out) {
#pragma omp parallel for schedule(static) if (n > 65536)
  for (int64_t i = 0; i < n; ++i) out[i] = (float)(scale * normal2(key, 2 * (uint64_t)i));
}

/* Router weights W_r [E x H] of a layer, N(0, 0.02). */
void syn_router_weights(uint64_t seed, int layer, int n_experts, int hidden, float* out) {
  syn_normal_f32(syn_key(seed, 2, (uint64_t)layer, 0, 0), 0.02, (int64_t)n_experts * hidden, out);
}

/* Activations of tokens [t0, t0+n) at one layer for one stream, N(0,1), [n x H]. */
void syn_activations(uint64_t seed, int layer, int stream, int64_t t0, int n, int hidden, float* out) {
  for (int i = 0; i < n; ++i)
    syn_normal_f32(syn_key(seed, 3, (uint64_t)layer, (uint64_t)stream, (uint64_t)(t0 + i)), 1.0, hidden,
                   out + (int64_t)i * hidden);
}

/* Seeded permutation pi_l: Zipf rank -> expert id (Fisher-Yates). */
void syn_permutation(uint64_t seed, int layer, int n, int32_t* perm) {
  uint64_t key = syn_key(seed, 5, (uint64_t)layer, 0, 0);
  for (int i = 0; i < n; ++i) perm[i] = i;
  for (int i = n - 1; i > 0; --i) {
    uint32_t r = (uint32_t)(draw(key, (uint64_t)i) >> 32);
    int j = (int)(((uint64_t)r * (uint64_t)(i + 1)) >> 32);
    int32_t t = perm[i];
    perm[i] = perm[j];
    perm[j] = t;
  }
}

/*
 * Route sets for n_tokens consecutive tokens of one stream at one layer.
 * With probability `reuse` a token repeats the previous token's set (same order);
 * otherwise k distinct Zipf ranks are drawn one after another without replacement,
 * P(rank r) proportional to (r+1)^-s over the ranks not yet drawn (s = 0: uniform),
 * and mapped to experts through pi_l.  out is [n_tokens x k] in draw order.
 */
int syn_routes(uint64_t seed, int layer, int stream, int n_experts, int top_k, int n_tokens,
               double zipf_s, double reuse, int32_t* out) {
  if (top_k <= 0 || top_k > n_experts || n_experts > 4096) return -1;
  int32_t perm[4096];
  double w[4096];
  unsigned char taken[4096];
  syn_permutation(seed, layer, n_experts, perm);
  for (int r = 0; r < n_experts; ++r) w[r] = pow((double)(r + 1), -zipf_s);
  uint64_t key = syn_key(seed, 4, (uint64_t)layer, (uint64_t)stream, 0);
  uint64_t ctr = 0;
  for (int t = 0; t < n_tokens; ++t) {
    int32_t* row = out + (int64_t)t * top_k;
    double u = unif(draw(key, ctr++));
    if (t > 0 && u < reuse) {
      memcpy(row, row - top_k, sizeof(int32_t) * (size_t)top_k);
      continue;
    }
    memset(taken, 0, (size_t)n_experts);
    for (int j = 0; j < top_k; ++j) {
      double total = 0.0;
      for (int r = 0; r < n_experts; ++r)
        if (!taken[r]) total += w[r];
      double target = unif(draw(key, ctr++)) * total;
      int pick = -1;
      double acc = 0.0;
      for (int r = 0; r < n_experts; ++r) {
        if (taken[r]) continue;
        pick = r;
        acc += w[r];
        if (target < acc) break;
      }
      taken[pick] = 1;
      row[j] = perm[pick];
    }
  }
  return 0;
}

/*
 * Speculative verification schedule (the workload of a verify-width study; no draft model):
 * verify step i checks K drafted tokens and the target accepts the first a_i of them, a_i =
 * the number of leading successes of independent trials that each succeed with probability
 * alpha (trial j of step i: value j of the stream of domain 6, step i).  The same schedule
 * serves every layer.  out[i] = a_i in [0, K].
 */
int syn_accepts(uint64_t seed, int stream, int n_steps, int K, double alpha, int32_t* out) {
  if (n_steps < 0 || K < 0 || !(alpha >= 0.0 && alpha <= 1.0)) return -1;
  for (int i = 0; i < n_steps; ++i) {
    const uint64_t key = syn_key(seed, 6, (uint64_t)stream, (uint64_t)i, 0);
    int a = 0;
    while (a < K && unif(draw(key, (uint64_t)a)) < alpha) ++a;
    out[i] = a;
  }
  return 0;
}
