/*
 * CPU oracle for the routed-expert step of one MoE decoder layer (MawForge,
 * arXiv 2607.09686).
 *
 * TEST INFRASTRUCTURE.  Only the test-suite, the package smoke check and the
 * benchmark's CPU-baseline leg load this library.  The product path never calls it and
 * shares no code, header or table with it.
 *
 * Plain and slow on purpose: every value is its definition written out, loop by loop,
 * in fp64.  The only parallelism is OpenMP over independent output rows, so each output
 * is computed by one thread in one fixed order and results do not depend on the thread
 * count.  Build with -ffp-contract=off (no fused multiply-add), which makes x86-64 and
 * aarch64 agree bit for bit.
 *
 * What it follows:
 *  - GGUF block formats (the format the paper serves, Background section): Q8_0
 *    weight = d * q, q int8; Q4_0 weight = d * (n - 8), n the 4-bit code, byte j of
 *    the 16 code bytes holding element j (low nibble) and element j+16 (high nibble);
 *    d an IEEE binary16 scale per 32 weights.
 *  - MoE routing (Background section; routed subset per token): logits z = W_r x
 *    (+ an optional per-token bias), the k largest logits chosen (ties to the lower
 *    expert id), weights = softmax over the chosen logits.
 *  - Expert FFN with separate gate, up and down tensors (section "Native Serving
 *    Path"): h = silu(W_gate x) * (W_up x), y_j = W_down h, silu(v) = v / (1 + e^-v);
 *    layer output y = sum_j g_j y_j.
 *  - Bounded per-layer slot cache (section "Native Serving Path": a miss materializes
 *    the expert block into an available slot and updates route-to-slot metadata):
 *    least-recently-used replacement, lowest free slot first.
 *  - Static budget check (section "Static Budget Check", L(p,n) = C + E(p) + K(n);
 *    reject when L exceeds the serving target) with the slot count of section
 *    "Native Serving Path" (slots from cache fraction, experts per layer and active
 *    experts per token).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_Q8_0 8
#define ORC_Q4_0 2

/* ---------- IEEE 754 binary16 -> value (sign, 5-bit exponent, 10-bit fraction) ---------- */
double orc_f16(uint16_t h) {
  int s = h >> 15, e = (h >> 10) & 0x1F, f = h & 0x3FF;
  double v;
  if (e == 0)
    v = ldexp((double)f, -24); /* subnormal: f * 2^-24 */
  else if (e == 31)
    v = f ? NAN : INFINITY;
  else
    v = ldexp((double)(1024 + f), e - 25); /* (1 + f/1024) * 2^(e-15) */
  return s ? -v : v;
}

static int block_bytes(int qtype) { return qtype == ORC_Q8_0 ? 34 : (qtype == ORC_Q4_0 ? 18 : 0); }

/* ---------- dequantise one row of `cols` weights (cols a multiple of 32) ---------- */
int orc_dequant_row(int qtype, const uint8_t* blocks, int cols, double* out) {
  int bb = block_bytes(qtype);
  if (!bb || cols % 32) return -1;
  for (int b = 0; b < cols / 32; ++b) {
    const uint8_t* blk = blocks + (size_t)b * bb;
    double d = orc_f16((uint16_t)(blk[0] | (blk[1] << 8)));
    if (qtype == ORC_Q8_0) {
      for (int i = 0; i < 32; ++i) out[32 * b + i] = d * (double)(int8_t)blk[2 + i];
    } else {
      for (int j = 0; j < 16; ++j) {
        int lo = blk[2 + j] & 0x0F, hi = blk[2 + j] >> 4;
        out[32 * b + j] = d * (double)(lo - 8);
        out[32 * b + j + 16] = d * (double)(hi - 8);
      }
    }
  }
  return 0;
}

/* bytes of one quantised tensor [rows x cols] */
static size_t tensor_bytes(int rows, int cols, int qtype) {
  return (size_t)rows * (size_t)(cols / 32) * (size_t)block_bytes(qtype);
}

uint64_t orc_payload_bytes(int hidden, int inter, int qtype) {
  return 2 * tensor_bytes(inter, hidden, qtype) + tensor_bytes(hidden, inter, qtype);
}

/* ---------- router: logits, top-k, softmax over the chosen ---------- */
/* z_e = fp32(sum_i W[e,i] x_i) computed with exact fp64 products and fp64 summation,
 * then + bias_e in fp32.  Chosen: the k largest z, ties to the lower id, listed in that
 * order.  g_j = exp(z_j - z_max) / sum_chosen exp(z - z_max) in fp64. */
static _Thread_local const float* g_sort_z; /* per thread: the oracle may be called from several threads */
static int cmp_desc(const void* a, const void* b) {
  int ia = *(const int*)a, ib = *(const int*)b;
  float za = g_sort_z[ia], zb = g_sort_z[ib];
  if (za > zb) return -1;
  if (za < zb) return 1;
  return ia < ib ? -1 : (ia > ib ? 1 : 0);
}

int orc_router(const float* x, const float* wr, const float* bias, int E, int H, int k, float* z,
               int32_t* idx, double* g) {
  if (k <= 0 || k > E) return -1;
  for (int e = 0; e < E; ++e) {
    double s = 0.0;
    for (int i = 0; i < H; ++i) s += (double)wr[(size_t)e * H + i] * (double)x[i];
    float zf = (float)s;
    if (bias) zf = zf + bias[e];
    z[e] = zf;
  }
  int* order = (int*)malloc(sizeof(int) * (size_t)E);
  if (!order) return -2;
  for (int e = 0; e < E; ++e) order[e] = e;
  g_sort_z = z;
  qsort(order, (size_t)E, sizeof(int), cmp_desc);
  double zmax = (double)z[order[0]], den = 0.0;
  for (int j = 0; j < k; ++j) den += exp((double)z[order[j]] - zmax);
  for (int j = 0; j < k; ++j) {
    idx[j] = order[j];
    g[j] = exp((double)z[order[j]] - zmax) / den;
  }
  free(order);
  return 0;
}

/* ---------- one expert's SwiGLU FFN on one token ---------- */
/* payload: gate [I x H], up [I x H], down [H x I] GGUF blocks back to back. */
int orc_expert_ffn(const uint8_t* payload, int qtype, int H, int I, const float* x, double* y,
                   double* h_out) {
  if (!block_bytes(qtype) || H % 32 || I % 32) return -1;
  const uint8_t* wg = payload;
  const uint8_t* wu = payload + tensor_bytes(I, H, qtype);
  const uint8_t* wd = payload + 2 * tensor_bytes(I, H, qtype);
  const size_t row_gu = tensor_bytes(1, H, qtype), row_d = tensor_bytes(1, I, qtype);
  double* h = (double*)malloc(sizeof(double) * (size_t)I);
  if (!h) return -2;
#pragma omp parallel
  {
    double* w = (double*)malloc(sizeof(double) * (size_t)(H > I ? H : I));
#pragma omp for schedule(static)
    for (int r = 0; r < I; ++r) {
      double gate = 0.0, up = 0.0;
      orc_dequant_row(qtype, wg + r * row_gu, H, w);
      for (int c = 0; c < H; ++c) gate += w[c] * (double)x[c];
      orc_dequant_row(qtype, wu + r * row_gu, H, w);
      for (int c = 0; c < H; ++c) up += w[c] * (double)x[c];
      h[r] = gate / (1.0 + exp(-gate)) * up;
    }
#pragma omp for schedule(static)
    for (int c = 0; c < H; ++c) {
      double acc = 0.0;
      orc_dequant_row(qtype, wd + c * row_d, I, w);
      for (int r = 0; r < I; ++r) acc += w[r] * h[r];
      y[c] = acc;
    }
    free(w);
  }
  if (h_out) memcpy(h_out, h, sizeof(double) * (size_t)I);
  free(h);
  return 0;
}

/* ---------- the layer: router + k expert FFNs + weighted combine, per token ---------- */
/* payloads[e] may be NULL for experts no token routes to (error -3 if one is needed).
 * bias is [T x E] or NULL.  y is rounded to fp32 once, at the end. */
int orc_layer(const uint8_t* const* payloads, int qtype, int E, int H, int I, int k, const float* wr,
              const float* bias, const float* x, int T, float* y, int32_t* idx, double* g) {
  float* z = (float*)malloc(sizeof(float) * (size_t)E);
  double* acc = (double*)malloc(sizeof(double) * (size_t)H);
  double* ye = (double*)malloc(sizeof(double) * (size_t)H);
  int rc = 0;
  if (!z || !acc || !ye) rc = -2;
  for (int t = 0; t < T && !rc; ++t) {
    const float* xt = x + (size_t)t * H;
    int32_t* it = idx + (size_t)t * k;
    double* gt = g + (size_t)t * k;
    rc = orc_router(xt, wr, bias ? bias + (size_t)t * E : NULL, E, H, k, z, it, gt);
    if (rc) break;
    for (int c = 0; c < H; ++c) acc[c] = 0.0;
    for (int j = 0; j < k && !rc; ++j) {
      if (!payloads[it[j]]) {
        rc = -3;
        break;
      }
      rc = orc_expert_ffn(payloads[it[j]], qtype, H, I, xt, ye, NULL);
      for (int c = 0; c < H && !rc; ++c) acc[c] += gt[j] * ye[c];
    }
    for (int c = 0; c < H; ++c) y[(size_t)t * H + c] = (float)acc[c];
  }
  free(z);
  free(acc);
  free(ye);
  return rc;
}

/* ---------- bounded LRU slot cache of one layer ---------- */
typedef struct orc_lru {
  int E, S;
  uint64_t payload, clock, accesses, hits, misses, evictions, bytes;
  int32_t* slot_of;   /* expert -> slot or -1 */
  int32_t* expert_of; /* slot -> expert or -1 */
  uint64_t* last_use; /* slot -> time of last access */
} orc_lru;

void orc_lru_free(orc_lru* c) {
  if (!c) return;
  free(c->slot_of);
  free(c->expert_of);
  free(c->last_use);
  free(c);
}

orc_lru* orc_lru_new(int E, int S, uint64_t payload) {
  if (E <= 0 || S <= 0 || S > E) return NULL;
  orc_lru* c = (orc_lru*)calloc(1, sizeof(orc_lru));
  if (!c) return NULL;
  c->E = E;
  c->S = S;
  c->payload = payload;
  c->slot_of = (int32_t*)malloc(sizeof(int32_t) * (size_t)E);
  c->expert_of = (int32_t*)malloc(sizeof(int32_t) * (size_t)S);
  c->last_use = (uint64_t*)calloc((size_t)S, sizeof(uint64_t));
  if (!c->slot_of || !c->expert_of || !c->last_use) {
    orc_lru_free(c);
    return NULL;
  }
  for (int e = 0; e < E; ++e) c->slot_of[e] = -1;
  for (int s = 0; s < S; ++s) c->expert_of[s] = -1;
  return c;
}

/* One step: the step's accesses are its distinct experts in (token, rank) first-occurrence
 * order; with order 1 and T > 1, the experts resident when the step starts come first (in
 * that order among themselves), then the others (likewise).  Each access: resident -> hit;
 * else miss into the lowest free slot, or, with no free slot, into the slot of the least
 * recently used expert, which is evicted.
 * Writes the access list (expert, slot after the access, hit bit); returns its length. */
int orc_lru_step(orc_lru* c, const int32_t* idx, int T, int k, int order, int32_t* uniq, int32_t* slot,
                 uint8_t* hit) {
  int U = 0;
  for (int p = 0; p < T * k; ++p) {
    int e = idx[p], seen = 0;
    if (e < 0 || e >= c->E) return -1;
    for (int u = 0; u < U; ++u)
      if (uniq[u] == e) seen = 1;
    if (!seen) uniq[U++] = e;
  }
  if (order == 1 && T > 1) { /* resident ones first, each group keeping its order */
    int32_t* first = (int32_t*)malloc(sizeof(int32_t) * (size_t)(U > 0 ? U : 1));
    if (!first) return -2;
    int n = 0;
    for (int u = 0; u < U; ++u)
      if (c->slot_of[uniq[u]] >= 0) first[n++] = uniq[u];
    for (int u = 0; u < U; ++u)
      if (c->slot_of[uniq[u]] < 0) first[n++] = uniq[u];
    memcpy(uniq, first, sizeof(int32_t) * (size_t)U);
    free(first);
  }
  for (int u = 0; u < U; ++u) {
    int e = uniq[u], s = c->slot_of[e];
    c->accesses++;
    if (s >= 0) {
      c->hits++;
      hit[u] = 1;
    } else {
      c->misses++;
      hit[u] = 0;
      for (int q = 0; q < c->S && s < 0; ++q)
        if (c->expert_of[q] < 0) s = q;
      if (s < 0) {
        s = 0;
        for (int q = 1; q < c->S; ++q)
          if (c->last_use[q] < c->last_use[s]) s = q;
        c->slot_of[c->expert_of[s]] = -1;
        c->evictions++;
      }
      c->expert_of[s] = e;
      c->slot_of[e] = s;
      c->bytes += c->payload;
    }
    c->last_use[s] = ++c->clock;
    slot[u] = s;
  }
  return U;
}

/* {accesses, hits, misses, evictions, bytes} */
void orc_lru_stats(const orc_lru* c, uint64_t* out) {
  out[0] = c->accesses;
  out[1] = c->hits;
  out[2] = c->misses;
  out[3] = c->evictions;
  out[4] = c->bytes;
}

int orc_lru_occupancy(const orc_lru* c) {
  int n = 0;
  for (int s = 0; s < c->S; ++s) n += c->expert_of[s] >= 0;
  return n;
}

/* slot -> expert map (length S) */
void orc_lru_slots(const orc_lru* c, int32_t* out) { memcpy(out, c->expert_of, sizeof(int32_t) * (size_t)c->S); }

/* ---------- static budget check ---------- */
/* S = max(k, floor(pct * E / 100)) (at most E); payload = canonical GGUF bytes of one
 * expert; E(p) = L * S * payload; lower = C + E(p) + K; accepted iff lower <= budget.
 * out = {S, payload, pool, lower, accepted}. */
int orc_plan(int L, int H, int E, int k, int I, int qtype, double pct, uint64_t budget, uint64_t common,
             uint64_t kv, uint64_t* out) {
  if (L <= 0 || E <= 0 || k <= 0 || k > E || !block_bytes(qtype) || H % 32 || I % 32 || pct < 0 || pct > 100)
    return -1;
  int S = (int)floor(pct * (double)E / 100.0 + 1e-9);
  if (S < k) S = k;
  if (S > E) S = E;
  uint64_t payload = orc_payload_bytes(H, I, qtype);
  uint64_t pool = (uint64_t)L * (uint64_t)S * payload;
  uint64_t lower = common + pool + kv;
  out[0] = (uint64_t)S;
  out[1] = payload;
  out[2] = pool;
  out[3] = lower;
  out[4] = lower <= budget;
  return 0;
}
