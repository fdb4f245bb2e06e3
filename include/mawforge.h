/*
 * mawforge.h — C ABI of the routed-expert step of one MoE decoder layer on one GB300.
 *
 * Method: MawForge, "Memory-Bounded Expert Materialization for Local Mixture-of-Experts
 * Inference" (arXiv 2607.09686).  Routed expert tensors live outside fast memory as
 * per-layer, per-expert payloads (section "Split-Pack Representation"); a bounded set
 * of per-layer slots holds the experts in use, and a miss copies the requested expert
 * block into an available slot and updates the route-to-slot metadata (section
 * "Native Serving Path"); a static check rejects a configuration whose lower bound
 * L(p, n) = C + E(p) + K(n) exceeds the serving target before anything is loaded
 * (section "Static Budget Check").
 *
 * Here the split-pack sits in pinned host memory, the slots in HBM, and one call of
 * mf_moe_forward runs, for one layer and T tokens, entirely in CUDA kernels:
 *   router logits + top-k + softmax over the chosen ->
 *   slot resolve (per-layer LRU, hit / miss / eviction / byte counters) ->
 *   materialisation of the missed payloads, pinned host -> HBM slot, on a side stream ->
 *   dequantising gate/up projections + SwiGLU -> down projection + router-weighted combine.
 *
 * Conventions for every entry point:
 *  - Return MF_OK (0) or a negative MF_E_* code; mf_strerror() names it.  A failing call
 *    changes no state the caller can observe, except MF_E_CUDA after a kernel launch
 *    failed (the context should then be destroyed).
 *  - Pointers documented "device" must be device memory of the context's GPU (or
 *    memory the GPU can address); "host" pointers are CPU memory.  The caller owns every
 *    buffer it passes; the library owns the pinned pack, the HBM slot pool, its scratch,
 *    its side stream and its events.
 *  - A context is not thread-safe: one host thread at a time per context.
 *  - Quantised weights use the GGUF block formats: Q8_0 = {binary16 d; int8 q[32]}
 *    (34 B, w = d*q); Q4_0 = {binary16 d; uint8 qs[16]} (18 B, byte j holds element j
 *    in its low nibble and element j+16 in its high nibble, w = d*(n-8)).
 */
#ifndef MAWFORGE_H
#define MAWFORGE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ---- */
#define MF_OK 0
#define MF_E_INVAL (-1)  /* an argument is out of range, NULL where required, or inconsistent */
#define MF_E_BUDGET (-2) /* the static plan rejected this configuration */
#define MF_E_OOM (-3)    /* pinned host or device allocation failed */
#define MF_E_CUDA (-4)   /* a CUDA runtime call or kernel launch failed */
#define MF_E_STATE (-5)  /* the call is not valid in the context's current state */
#define MF_E_TIMEOUT (-6) /* a bounded wait inside a kernel gave up (reported by mf_check) */
#define MF_E_IO (-7)      /* reading a split-pack file failed (reported by mf_check) */

/* ---- quantisation types (GGUF type ids) ---- */
#define MF_Q4_0 2
#define MF_Q8_0 8

/* Access orders of a step with several tokens (mf_access_order). */
#define MF_ORDER_FIRST_OCCURRENCE 0 /* distinct experts in (token, rank) first-occurrence order */
#define MF_ORDER_RESIDENT_FIRST 1   /* the experts resident when the step starts first, then the rest */

/* Shape of the routed-expert part of a model.  Each expert is a SwiGLU FFN with separate
 * gate [inter x hidden], up [inter x hidden] and down [hidden x inter] tensors.
 * Requirements: hidden and inter multiples of 32; 1 <= top_k <= 8; top_k <= n_experts <= 1024. */
typedef struct mf_model {
  int32_t n_layers, hidden, n_experts, top_k, inter, qtype;
} mf_model_t;

/* Static-plan request (section "Static Budget Check").
 * cache_pct: expert-cache size as a percentage p of the experts of each layer (0..100).
 * budget_bytes: the serving target; common_bytes: resident common tensors C;
 * kv_bytes: K(n); max_tokens: the largest T a single mf_moe_forward call will pass. */
typedef struct mf_plan_req {
  double cache_pct;
  uint64_t budget_bytes, common_bytes, kv_bytes;
  int32_t max_tokens, reserved;
} mf_plan_req_t;

/* Static-plan result.
 * slots_per_layer S = max(top_k, floor(p * n_experts / 100)), at most n_experts;
 * payload_bytes: canonical GGUF bytes of one expert (gate + up + down);
 * pool_bytes E(p) = n_layers * S * payload_bytes;
 * lower_bound_bytes L = C + E(p) + K; accepted = (L <= budget);
 * overhead_bytes O: this library's device scratch and slot-table bytes for max_tokens;
 * footprint_bytes F = L + O (section "Static Budget Check"). */
typedef struct mf_plan {
  int32_t accepted, slots_per_layer;
  uint64_t payload_bytes, pool_bytes, lower_bound_bytes, overhead_bytes, footprint_bytes;
  int32_t max_tokens, reserved;
} mf_plan_t;

/* Cache counters of one layer, or summed over layers (section "Native Serving Path";
 * the CLI of the paper reports hit rate and materialised expert bytes).
 * accesses = hits + misses; bytes_materialized = misses * payload_bytes. */
typedef struct mf_stats {
  uint64_t accesses, hits, misses, evictions, bytes_materialized;
} mf_stats_t;

typedef struct mf_ctx mf_ctx_t;

/* Canonical GGUF bytes of one expert payload.  Host only. */
int mf_payload_bytes(const mf_model_t* model, uint64_t* out);

/* One candidate cache size of mf_tune_cache. */
typedef struct mf_tune_point {
  double cache_pct;                 /* the candidate p (copied from the request) */
  int32_t accepted, slots_per_layer; /* mf_plan's decision and S for p */
  uint64_t pool_bytes, footprint_bytes;
  uint64_t accesses, hits, misses;  /* the trace replayed through per-layer caches of S slots */
  uint64_t bytes_materialized;      /* misses * payload_bytes */
  double predicted_s;               /* n_tokens * t_token_s + misses * t_miss_s */
  double predicted_tokens_per_s;    /* n_tokens / predicted_s (0 when predicted_s is 0) */
} mf_tune_point_t;

/* Cache-size tuner (section "Throughput Model": T(p) = tokens / (compute_time +
 * materialization_time(p) + pressure_penalty(F)); Discussion, "Cache Hit Rate Is an Incomplete
 * Objective": choose the cache point that minimises end-to-end latency under the memory budget,
 * not the one that maximises hit rate).  Host only, no GPU needed.
 *   routes    host int32 [n_layers][n_tokens][top_k]: a route trace (expert ids in [0,
 *             n_experts), each token's in the router's rank order, as idx_out returns them: the
 *             order the cache sees), replayed layer by layer in steps of T consecutive tokens
 *             (the last step may be shorter), with the library's cache semantics: per step the
 *             distinct experts in the given access order (MF_ORDER_*), least-recently-used
 *             replacement
 *   t_token_s measured seconds per token with every expert resident (all layers);
 *   t_miss_s  measured seconds per materialised payload (the link's share of a miss)
 *   pcts      host [n] candidate cache percentages; req supplies the other plan inputs
 *   out       host [n] results, in the order of pcts; *best = the accepted candidate with the
 *             highest predicted rate (ties: the smaller pool, then the earlier candidate), or -1
 * The pressure term is zero: on a GB300 the slot pool is dedicated HBM, so a plan inside the
 * static budget pages nothing.  MF_E_INVAL for NULL pointers, n < 1, n_tokens < 1, T < 1, an
 * expert id out of range, negative or non-finite times, an unknown order or an invalid p;
 * MF_E_BUDGET (with out and *best = -1 filled) when no candidate is accepted. */
int mf_tune_cache(const mf_model_t* model, const mf_plan_req_t* req, const int32_t* routes, int n_tokens, int T,
                  int order, double t_token_s, double t_miss_s, const double* pcts, int n, mf_tune_point_t* out,
                  int* best);

/* Static budget check (section "Static Budget Check").  Host-only arithmetic, no GPU
 * needed.  Fills *out even when rejecting; returns MF_E_BUDGET if L > budget. */
int mf_plan(const mf_model_t* model, const mf_plan_req_t* req, mf_plan_t* out);

/* Create a context on CUDA device `device` (section "Split-Pack Representation": routed expert
 * tensors are held outside fast memory as per-layer, per-expert payloads, and the runtime
 * materialises only the experts a step needs; section "Native Serving Path": bounded per-layer
 * slots).  Allocates the pinned host pack (n_layers * n_experts payloads: the split-pack), the
 * HBM slot pool (n_layers * S payloads), the slot table and the scratch for plan->max_tokens.
 * Refuses a rejected plan (MF_E_BUDGET); MF_E_INVAL for an invalid model or a plan that does not
 * belong to it; MF_E_OOM when an allocation fails (nothing is left allocated).  The pack is
 * empty: fill it with mf_pack_put before the first mf_moe_forward (MF_E_STATE until then). */
int mf_create(mf_ctx_t** out, const mf_model_t* model, const mf_plan_t* plan, int device);

/* Copy one expert's canonical GGUF payload (host memory, `bytes` must equal payload_bytes)
 * into its place in the pinned split-pack (section "Split-Pack Representation": one payload per
 * (layer, expert), gate, up and down tensors together), repacked into row records so that
 * quantised codes and scales are 16-byte aligned and the rows a kernel computes together are
 * contiguous (the same bytes, regrouped; accounting stays at payload_bytes).  The caller may free
 * `payload` when the call returns.  MF_E_INVAL for a NULL payload, a layer or expert out of range
 * or a wrong size.  Host only, synchronous; calls for distinct (layer, expert) pairs may run
 * concurrently from several host threads. */
int mf_pack_put(mf_ctx_t* ctx, int layer, int expert, const void* payload, uint64_t bytes);

/* Write the context's split-pack to a file (section "Split-Pack Representation": the expert
 * payloads in one pack file with an index of layer, expert, offset, byte count and digest, so the
 * runtime can address one expert block without reading unrelated weights).  Layout: a 4096-byte
 * header (magic "MFSPLIT1", version 1, the model, payload bytes, slot-layout bytes, record bytes,
 * index and record offsets), the index (one 32-byte entry per (layer, expert), layer-major: layer,
 * expert, record offset, payload bytes, 64-bit FNV-1a digest of the record's bytes), then one
 * record per payload in the pack's slot layout, each padded to a multiple of 4096 bytes.  Every
 * payload must have been put (MF_E_STATE otherwise, and for a file-backed context); MF_E_INVAL
 * for a NULL path or when the file cannot be written (a partial file is removed).  Host only. */
int mf_pack_save(mf_ctx_t* ctx, const char* path);

/* As mf_create, but the split-pack is the file `path` written by mf_pack_save (the disk tier:
 * the model stays a disk object; section "Split-Pack Representation", and the Introduction's
 * memory hierarchy of disk, memory and slots).  No pinned pack is allocated: misses are still
 * decided on the GPU, and after the kernels that decide them a host function on the call's stream
 * reads the missed records from the file (all of the call's misses, or a wave's, in parallel
 * 1 MiB reads, unbuffered where the file system allows it) into pinned staging of max(top_k, S)
 * records, from which the kernels copy them into their slots over the CPU-GPU link.  Calls are
 * stream-ordered as usual and may be captured into CUDA graphs (the reads become host nodes).
 * MF_E_INVAL if the file is missing, truncated, or its header or index do not match the model;
 * MF_E_OOM if the staging cannot be allocated.  mf_pack_put on such a context returns
 * MF_E_STATE.  A failed read is reported by mf_check as MF_E_IO. */
int mf_create_from_file(mf_ctx_t** out, const mf_model_t* model, const mf_plan_t* plan, const char* path,
                        int device);

/* Reads of a file-backed context since its creation: payload records read, bytes read and the
 * seconds the reads took (summed over calls, host clock).  MF_E_INVAL for a context without a
 * file.  Host only; counts only calls the stream has reached. */
int mf_pack_file_stats(mf_ctx_t* ctx, uint64_t* reads, uint64_t* bytes, double* seconds);

/* 1 if the file-backed context reads its file unbuffered (O_DIRECT), 0 if through the page cache,
 * MF_E_INVAL for a context without a file. */
int mf_pack_file_direct(mf_ctx_t* ctx);

/* mf_create followed by mf_pack_put of payloads[layer * n_experts + expert] (host
 * pointers, each payload_bytes long) for every layer and expert: the whole split-pack loaded
 * (section "Split-Pack Representation").  MF_E_INVAL if any pointer is NULL; on any failure
 * nothing is left allocated and *out is NULL. */
int mf_load_pack(mf_ctx_t** out, const mf_model_t* model, const mf_plan_t* plan,
                 const void* const* payloads, int device);

/* One routed-expert step of layer `layer` for T tokens, stream-ordered on `stream`
 * (a cudaStream_t; NULL = the legacy default stream).
 *   x          device float [T][hidden]      token activations
 *   router_w   device float [n_experts][hidden]  router weights W_r
 *   logit_bias device float [T][n_experts] or NULL, added to the logits in fp32
 *   y          device float [T][hidden]      output: sum_j g_j * FFN_{e_j}(x_t)
 *   idx_out    device int32 [T][top_k] or NULL: chosen experts, largest logit first
 *              (ties to the lower expert id)
 *   w_out      device float [T][top_k] or NULL: softmax of the chosen logits
 * Each layer's cache is one LRU over that layer's calls, in call order: calls for one
 * layer must be issued in token order.  Within a call the accesses are the distinct
 * experts of the T tokens in (token, rank) first-occurrence order; when there are more
 * than S of them they are processed in waves of S.  0 <= T <= plan max_tokens; T = 0
 * does nothing.  Inputs must be finite.  Returns after enqueueing (no host sync). */
int mf_moe_forward(mf_ctx_t* ctx, int layer, const float* x, const float* router_w,
                   const float* logit_bias, int T, float* y, int32_t* idx_out, float* w_out,
                   void* stream);

/* Calls of mf_moe_forward with T >= min_tokens run each wave's expert FFN as tcgen05 grouped
 * GEMMs (section "Native Serving Path"'s expert FFN, batched over the tokens each expert
 * serves, as for a prefill chunk): per (expert, 128 assignments, 128 weight rows) the
 * dequantised Q8_0 / Q4_0 weights and the activations, each split into bf16 hi + lo, are
 * multiplied on the tensor cores with fp32 accumulation (hi*hi + hi*lo + lo*hi).  Smaller T
 * use the dequantising GEMV kernels.  The default is 256 when the plan's max_tokens >= 256,
 * else 0 (off).  min_tokens = 0 disables the GEMM path; otherwise it must be >= 2, the plan's
 * max_tokens >= 2 and hidden and inter multiples of 128 (MF_E_INVAL otherwise).  Enabling it
 * on a context created with max_tokens < 256 allocates its operand tiles here:
 * (T k / 128 + min(E, T k)) * 128 * (hidden + inter) * 4 bytes for T = max_tokens (MF_E_OOM
 * if that fails; MF_E_CUDA if the driver cannot describe the slot pool to the copy engine).
 * Host only; applies to calls issued afterwards. */
int mf_prefill_threshold(mf_ctx_t* ctx, int min_tokens);

/* Order in which a call with T > 1 presents its distinct experts to the layer's cache
 * (section "Native Serving Path": the cache is consulted per routed expert; the paper does not
 * order a batched step's accesses).  MF_ORDER_FIRST_OCCURRENCE (the default): (token, rank)
 * first-occurrence order.  MF_ORDER_RESIDENT_FIRST: the experts that are resident when the
 * call starts come first (in first-occurrence order among themselves), then the others (in
 * first-occurrence order): every one of them hits, whereas in first-occurrence order an early
 * miss can evict an expert the same step needs later.  Calls with T = 1 keep first-occurrence
 * order whatever is set (the order applies to calls with T > 1 only).  Waves,
 * counters, traces and outputs follow the chosen order.  MF_E_INVAL for any other value.  Host
 * only; applies to calls issued afterwards. */
int mf_access_order(mf_ctx_t* ctx, int order);

/* As mf_moe_forward, with x, logit_bias, y, idx_out and w_out in HOST memory.  Pageable
 * buffers: x and the bias are staged into the context's device buffers and the outputs copied
 * back, all on `stream`.  Pinned buffers (cudaHostAlloc / cudaHostRegister) with T = 1: no copy
 * steps -- the kernels read x and the bias and write y over the CPU-GPU link.  The host buffers
 * must stay valid until the stream reaches the end of the call (synchronise before reading y). */
int mf_moe_forward_host(mf_ctx_t* ctx, int layer, const float* x, const float* router_w,
                        const float* logit_bias, int T, float* y, int32_t* idx_out, float* w_out,
                        void* stream);

/* Cache counters of `layer`, or summed over all layers when layer = -1.  Synchronises
 * the context's device work first.  reset != 0 zeroes the counters read. */
int mf_stats(mf_ctx_t* ctx, int layer, mf_stats_t* out, int reset);

/* Make every layer's cache cold and zero all counters; if slots_per_layer > 0, also set
 * the number of slots in use per layer (top_k <= slots_per_layer <= the planned S).
 * Stream-ordered on `stream`. */
int mf_reset(mf_ctx_t* ctx, int slots_per_layer, void* stream);

/* The access record of the most recent mf_moe_forward call of `layer`: for each access
 * u < *n, the expert, its slot after the access and whether it hit.  Host arrays of
 * `cap` entries; synchronises the context's device work first. */
int mf_trace(mf_ctx_t* ctx, int layer, int32_t* experts, int32_t* slots, uint8_t* hits, int cap,
             int* n);

/* Per-kernel timing with CUDA events recorded on the stream each kernel runs on.
 * class_mask selects the kernel classes timed (bit i: 0 router, 1 resolve, 2 materialise,
 * 3 gate/up+SwiGLU, 4 down+combine, 5 prefill grouped GEMMs, 6 one-token expert FFN (gate/up,
 * SwiGLU, down and combine in one launch); 0 stops timing); each call clears
 * earlier records.  mf_timing_read synchronises and writes for each class the summed
 * milliseconds and the number of timed launches into ms[7] and launches[7].  Calls captured
 * into a CUDA graph while timing is on capture their event records as graph nodes; after each
 * replay mf_timing_read reports that replay. */
int mf_timing(mf_ctx_t* ctx, unsigned class_mask);
int mf_timing_read(mf_ctx_t* ctx, double* ms, int64_t* launches);

/* Synchronise the device and report whether any kernel of this context gave up a bounded
 * wait since the last check (MF_E_TIMEOUT), clearing the record.  Kernels never spin without a
 * limit: a pipeline stage that is not filled or released, or a block whose partner blocks do not
 * publish their part, within the time limit (mf_wait_limit) makes the kernel record the failure
 * and return.  After MF_E_TIMEOUT the outputs of the calls since the last check are unreliable,
 * and so may be the contents of slots materialised by them: call mf_reset before relying on the
 * cache again.  The context itself stays usable. */
int mf_check(mf_ctx_t* ctx);

/* Time limit, in seconds (1e-6 .. 60), of every bounded wait inside this context's kernels
 * (default 1 s): a wait that has not completed after that long gives up as described under
 * mf_check.  MF_E_INVAL outside the range.  Host only; applies to calls issued afterwards
 * (calls already captured into a CUDA graph keep the limit they were captured with). */
int mf_wait_limit(mf_ctx_t* ctx, double seconds);

/* Test hold for the failure path (no counterpart in the paper).  hold = 1: the producer warp of
 * the one-token expert FFN kernel issues none of its HBM copies, so the stages its consumers wait
 * for are never filled: their bounded waits run out after the wait limit, the kernel records the
 * failure and returns with nothing in flight, and mf_check reports MF_E_TIMEOUT.  Nothing faults
 * or hangs.  Calls whose experts all hit move no other bytes, so the cache stays consistent;
 * hold = 0 (the default) restores normal operation.  MF_E_INVAL for other values.  Host only;
 * applies to calls issued afterwards. */
int mf_test_hold(mf_ctx_t* ctx, int hold);

/* One-token expert FFN with no allocation at all (the paper has no counterpart: it is a
 * convenience of this library).  Callers that cannot allocate device memory — code running
 * while a CUDA graph is being captured under a no-allocation policy, latency-critical threads
 * that must not take cudaMalloc's implicit device synchronisation, or plugins confined to a
 * device-memory budget reserved by their host process — can still compute
 *   y = sum_j g[j] * down_j( silu(gate_j x) * (up_j x) ),   j < model->top_k,
 * from expert weights they already hold, without creating a context.  It runs the kernels of
 * a one-token mf_moe_forward; their intermediate h and index tables live in a file-scope
 * device array of 128 KiB + 256 B, which every GPU that loads this library holds until the
 * process exits.
 *   model    hidden, inter, top_k (<= 8) and qtype are used; top_k * inter must be <= 32768
 *            (else MF_E_INVAL: the static scratch is sized for that)
 *   experts  device, 16-byte aligned: top_k expert slots back to back, slot j = expert j, each
 *            `stride` bytes in this layout (Q = bytes of codes per row: hidden (Q8_0) or
 *            hidden/2 (Q4_0) for gate/up rows, inter or inter/2 for down rows; nb = weights/32):
 *              rs_gu = round16(2*Q_gu + round16(2*nb_gu) + 2*nb_gu), rs_d = round16(Q_d + 2*nb_d),
 *              d_off = round256(inter * rs_gu), stride = round256(d_off + hidden * rs_d);
 *              gate/up record r at r*rs_gu: [gate codes row r][up codes row r]
 *                [gate scales row r (nb_gu binary16), zero padding to a multiple of 16 bytes]
 *                [up scales row r], zero padding;
 *              down record c at d_off + c*rs_d: [down codes row c][down scales row c];
 *              codes in GGUF block order, Q8_0 codes stored as q + 128 (unsigned byte)
 *   g        device float [top_k] weights of the experts; x device float [hidden], 16-byte
 *            aligned; y device float [hidden] output
 * Stream-ordered on `stream`; returns after enqueueing.  The first call on each device sets up
 * that device (it reads the array's device address and writes its constant tables): make that
 * first call before any stream capture; host threads that make their first call at the same time
 * take turns.  All calls on a device share the array, so calls whose kernels overlap on the GPU
 * (other streams, other host threads) race on it: serialise them.  Nothing in the array needs
 * clearing between calls; h is fully rewritten by each call.  A bounded wait that gives up is
 * reported by mf_expert_ffn_noalloc_check. */
int mf_expert_ffn_noalloc(const mf_model_t* model, const void* experts, const float* g, const float* x,
                          float* y, void* stream);

/* Failure report of mf_expert_ffn_noalloc on the current device (its kernels' bounded waits give
 * up after 1 s and record that in the same static array): synchronises the device and returns
 * MF_E_TIMEOUT if a wait gave up since the last check, clearing the record, else MF_OK (also
 * when no call has run on the device).  Allocates nothing; MF_E_CUDA if the device cannot be
 * read. */
int mf_expert_ffn_noalloc_check(void);

/* Release everything the context owns (synchronises its streams first). NULL is a no-op. */
void mf_destroy(mf_ctx_t* ctx);

/* Static string naming a status code. */
const char* mf_strerror(int status);

/* Text of the last CUDA error seen by this library in the calling thread ("" if none). */
const char* mf_last_cuda_error(void);

#ifdef __cplusplus
}
#endif

#endif /* MAWFORGE_H */
