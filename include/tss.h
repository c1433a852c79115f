/*
 * tss.h -- C ABI of the GB300 (sm_103a) TSS target-side verification library (libtss.so).
 *
 * The library runs one verification step of speculative decoding on the *target* model, as the
 * paper "TSS: Target-Side Sparsification for Speculative Decoding in Domain-Specific Large
 * Language Models" states the problem:
 *
 *   - Sec. "Problem Formulation": the target has L blocks; a skip configuration S_d is a subset of
 *     them, and S_d = {} is the dense verifier.  The draft proposes candidate tokens that the
 *     target scores in parallel.
 *   - Sec. "Domain-to-Configuration Mapping": Phi maps each supported domain to its skip set;
 *     one complete target model serves every domain's sparse path.
 *   - Sec. "Domain-Aware Skip Controller", first equation: S(x) = Phi(d(x)) for a supported
 *     domain and the empty set otherwise, fixed for the whole request; second equation:
 *     h_{l+1} = f_l(h_l) for l not in S(x), h_{l+1} = h_l for l in S(x).
 *   - Sec. "Models and speculative decoding methods": the accept/reject rule is the base
 *     method's, unchanged (greedy at temperature 0; speculative sampling otherwise).
 *
 * f_l is a LLaMA block (App. "Models"): RMSNorm, rotary multi-head attention (rotate-half
 * pairing), SwiGLU MLP.  Weights are bf16; residual and accumulation are fp32.  On the default
 * (persistent) path every GEMM activation keeps about 16 significant bits (it is fed to the bf16
 * tensor cores as two parts, bf16(x) and bf16(x - bf16(x))), attention scores use fp16 q and k,
 * and the attention probabilities enter P.V as two bf16 parts; the new K/V rows are stored in
 * bf16.
 *
 * Conventions for every entry point:
 *   - Pointers are plain addresses.  "device" means CUDA device memory of the current device,
 *     "host" means host memory (pinned memory recommended where copies are asynchronous).
 *   - A stream is a cudaStream_t passed as void* (NULL = the legacy default stream).
 *   - Every call returns tss_status.  Errors the host can detect are reported before any work is
 *     enqueued and leave all caller buffers untouched; tss_last_error() then gives a message.
 *   - Kernels never trap.  A check that fails on the device records a code in a device status
 *     word and the kernel continues with a safe value; the code is reported by
 *     tss_sync_status() (TSS_ERR_DEVICE_CHECK or TSS_ERR_TIMEOUT).
 *   - Layer indices are 0-based: bit l of a skip mask names layer l.
 */
#ifndef TSS_H
#define TSS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int tss_status;
#define TSS_OK 0
#define TSS_ERR_INVALID_ARG 1     /* an argument failed host-side validation */
#define TSS_ERR_OUT_OF_MEMORY 2   /* a device allocation at tss_create failed */
#define TSS_ERR_KV_CAPACITY 3     /* ctx_len + n_nodes exceeds the KV cache capacity */
#define TSS_ERR_CUDA 4            /* a CUDA runtime/driver call failed */
#define TSS_ERR_UNSUPPORTED_ARCH 5 /* model shape or GPU (not sm_103) unsupported */
#define TSS_ERR_TIMEOUT 6         /* a bounded device-side wait gave up */
#define TSS_ERR_DEVICE_CHECK 7    /* a device-side input check failed (e.g. token id range) */

#define TSS_MODE_GREEDY 0 /* temperature 0: argmax acceptance, chain or tree */
#define TSS_MODE_SAMPLE 1 /* speculative sampling at temperature > 0, chain drafts */

typedef struct tss_ctx tss_ctx; /* opaque; owns repacked weights and all workspaces */

/* Model shape and capacity limits.
 *   n_layers <= 64; head_dim 64 or 128; d_model = n_heads * head_dim, a multiple of 128 and at
 *   most 8192.
 *   max_batch: requests per verify (<= 64).  max_rows: total draft-block rows per verify
 *   (<= 256).  max_nodes: rows per request, root included (<= 128; a step with a block of more than 64 rows runs
 *   each layer's attention as a separate kernel, the persistent kernel's in-kernel attention taking
 *   blocks of up to 64).  max_domains: size of the domain table Phi.
 *   max_positions: RoPE positions must be < max_positions. */
typedef struct {
  int n_layers, d_model, n_heads, head_dim, d_mlp, vocab;
  float rms_eps, rope_theta;
  int max_batch, max_rows, max_nodes, max_domains, max_positions;
} tss_arch;

/* Caller-owned bf16 weights in device memory, row-major [out][in] (PyTorch nn.Linear layout).
 * Per-layer fields are HOST arrays of n_layers device pointers.
 *   embed [vocab][d_model], lm_head [vocab][d_model], final_norm / attn_norm / mlp_norm
 *   [d_model], wq wk wv wo [d_model][d_model], w_gate w_up [d_mlp][d_model],
 *   w_down [d_model][d_mlp].
 * tss_create copies and repacks them; the caller may free its buffers when it returns. */
typedef struct {
  const void* embed;
  const void* lm_head;
  const void* final_norm;
  const void* const* attn_norm;
  const void* const* wq;
  const void* const* wk;
  const void* const* wv;
  const void* const* wo;
  const void* const* mlp_norm;
  const void* const* w_gate;
  const void* const* w_up;
  const void* const* w_down;
} tss_weights;

/* One verification step for n_req requests.  Rows are the requests' draft blocks concatenated
 * in request order; M = sum(n_nodes).  Row 0 of each block is the root (the last committed
 * token, whose KV is not yet cached); rows 1.. are draft nodes.
 *   n_nodes, ctx_len, domain_id, kv_slot, parent_idx, positions: HOST arrays.
 *     n_nodes[b]   in [1, max_nodes] (max_nodes <= 128)
 *     ctx_len[b]   tokens of request b already in its KV cache (>= 0)
 *     domain_id[b] key into Phi; an id never configured (or out of range) means dense
 *     kv_slot[b]   cache slot of request b (distinct); NULL means slot b
 *     parent_idx[M] request-local parent: -1 for row 0 only, otherwise in [0, own index)
 *                  (a chain is i-1)
 *     positions[M] RoPE positions; NULL means ctx_len + depth, otherwise must equal it
 *   tokens[M] (int32), draft_probs, uniforms: DEVICE arrays, or HOST arrays when io_host != 0.
 *     draft_probs (SAMPLE): [M][vocab] fp32; row i is the draft distribution that proposed the
 *       token of row i (row 0 unused).
 *     uniforms (SAMPLE, optional): [n_req][uniform_stride] fp32 in [0,1); for a chain of k
 *       drafts slot i-1 is the accept test of draft i (i=1..k) and slot k+i-1 the residual draw
 *       at draft i or the bonus draw (i=k+1).  NULL: the library draws them with
 *       Philox4x32-10, key (seed lo, seed hi), counter (slot, request, offset lo, offset hi),
 *       u = (first word >> 8) * 2^-24.
 *   io_host != 0: the inputs above and every result array are HOST pointers; the library
 *     copies them in and out on the stream (results are valid after the stream synchronises). */
typedef struct {
  int n_req;
  const int32_t* n_nodes;
  const int32_t* ctx_len;
  const int32_t* domain_id;
  const int32_t* kv_slot;
  const int32_t* parent_idx;
  const int32_t* positions;
  const int32_t* tokens;
  int mode;
  float temperature;
  const float* draft_probs;
  const float* uniforms;
  int uniform_stride;
  uint64_t philox_seed;
  uint64_t philox_offset;
  int io_host;
} tss_verify_batch;

/* Caller-owned KV cache.  layer is a HOST array of n_layers device pointers; layer l points to a
 * bf16 buffer [n_slots][2][n_heads][cap][head_dim] (K then V).  An entry may be NULL for a
 * layer that no request of a batch runs.  The library reads rows [0, ctx_len) and writes rows
 * [ctx_len, ctx_len + n_nodes) of every layer a request runs, and never touches the layers it
 * skips. */
typedef struct {
  void* const* layer;
  int n_slots;
  int cap;
} tss_kv_cache;

/* Caller-owned results (DEVICE arrays, or HOST arrays when io_host != 0).
 *   accept_len[n_req]       accepted draft tokens a
 *   bonus[n_req]            token emitted after the accepted ones
 *   path[n_req][path_stride] request-local rows of the accepted path: path[0] = 0 (root),
 *                           path[1..a] the accepted nodes, -1 after; path_stride > max depth
 *   new_ctx_len[n_req]      ctx_len + 1 + a (root and accepted drafts are now cached)
 *   logits[M][vocab]        fp32 target logits of every row, or NULL */
typedef struct {
  int32_t* accept_len;
  int32_t* bonus;
  int32_t* path;
  int path_stride;
  int32_t* new_ctx_len;
  float* logits;
} tss_verify_result;

/* Build a verifier on the current CUDA device (must be sm_103).  Copies and repacks the weights
 * into library-owned device memory, allocates every workspace for the limits in *arch, and
 * returns an opaque context.  Errors: INVALID_ARG, UNSUPPORTED_ARCH, OUT_OF_MEMORY, CUDA; on
 * error everything allocated so far is freed and *out is NULL.  For failure injection, the
 * environment variable TSS_ALLOC_LIMIT_BYTES=N makes the allocations fail with OUT_OF_MEMORY
 * once they would pass N bytes.  TSS_WAIT_LIMIT_MS=N (1..600000, default 2000) bounds every
 * device-side wait of the persistent kernel (see tss_inject_timeout); the tcgen05 attention's
 * waits are bounded by 2 s. */
tss_status tss_create(const tss_weights* weights, const tss_arch* arch, tss_ctx** out);

/* Phi(domain_id) = the set of layers whose bit is set in layer_bitmask (bit l = skip layer l;
 * 0 = dense).  Sec. "Domain-to-Configuration Mapping".  Bits >= n_layers must be clear.
 * Host-only and immediate: no device work and no wait.  tss_verify looks up each request's
 * S(x) = Phi(d(x)) when it is called and passes the result to the device with the step, so a
 * verify already enqueued runs under the map it was enqueued with and later verifies see the
 * change.  domain_id in [0, max_domains).  Not thread-safe against concurrent calls on the same
 * context (like every call taking a tss_ctx*). */
tss_status tss_set_skip_config(tss_ctx* ctx, int domain_id, uint64_t layer_bitmask);

/* Remove domain_id from Phi: its requests then run the dense path (unsupported domain).
 * Host-only and immediate, as tss_set_skip_config. */
tss_status tss_clear_skip_config(tss_ctx* ctx, int domain_id);

/* Sparsity ratio R_d = |S_d| / L of a configured domain (0 for an unconfigured one), and the
 * number of layers the union of a batch's skip sets leaves active.  Host-only queries. */
tss_status tss_sparsity_ratio(const tss_ctx* ctx, int domain_id, double* out);
tss_status tss_active_layer_count(const tss_ctx* ctx, const tss_verify_batch* batch, int* out);

/* Bytes a verification step must move through HBM, the numerator of its roofline.  On this
 * memory-bound path the verification cost C_d(S) of Sec. "Problem Formulation" is proportional
 * to it, so an offline search over skip sets can rank candidates without running them.
 *   weights  = |union of the requests' active layers| x 2(4 d^2 + 3 d d_mlp)  +  vocab x d x 2
 *              (every active layer's weights and the LM head, read once per step);
 *   kv_read  = sum over requests of ctx_len x (layers it runs) x 4 d   (its context K and V);
 *   kv_write = sum over requests of n_nodes x (layers it runs) x 4 d   (the rows it appends);
 *   total    = weights + kv_read + kv_write; active_union = the size of the union.
 * masks[n_req] (bit l set = request skips layer l, i.e. S(x)), ctx_len[n_req] and
 * n_nodes[n_req] are HOST arrays.  Pure host arithmetic: no context and no CUDA call.  Errors:
 * INVALID_ARG (NULL argument, n_req < 1, a mask bit >= n_layers, a negative length). */
typedef struct {
  uint64_t weights, kv_read, kv_write, total;
  int active_union;
} tss_step_bytes;
tss_status tss_estimate_step_bytes(const tss_arch* arch, int n_req, const uint64_t* masks, const int32_t* ctx_len,
                                   const int32_t* n_nodes, tss_step_bytes* out);

/* Shared-memory plan of the persistent verify kernel for a step of n_req requests with n_rows
 * draft-block rows in all, whose longest request spans max_keys keys (context + block), on a
 * GPU with num_sms SMs, under the default switches: fits = 1 when the plan fits the 227 KiB a
 * block may use (then tss_verify runs the step; otherwise it returns TSS_ERR_UNSUPPORTED_ARCH),
 * with the weight k-blocks per ring stage, the ring stages, the attention's key splits and the
 * dynamic shared memory of one block.  Pure host arithmetic: no context and no CUDA call.
 * Errors: INVALID_ARG (NULL argument, head_dim not 64/128, n_req outside [1, 64], n_rows
 * outside [n_req, 256], max_keys or num_sms < 1). */
typedef struct {
  int fits, kps, stages, attn_splits;
  uint64_t smem_bytes;
} tss_persistent_plan_info;
tss_status tss_persistent_plan(const tss_arch* arch, int n_req, int n_rows, int max_keys, int num_sms,
                               tss_persistent_plan_info* out);

/* One verification step, enqueued on `stream`: skip controller (per-request S(x), union of
 * active layers, per-layer compacted row lists) -> embedding -> for every layer in the union:
 * RMSNorm+QKV GEMM with RoPE and KV append, split-KV attention with the chain/tree mask,
 * O projection, RMSNorm+SwiGLU MLP -> final norm + LM head with fused argmax -> acceptance
 * (greedy walk or speculative sampling) -> KV compaction of the accepted path.  A skipped layer
 * gets no launch, reads no weight byte and no KV row.  Asynchronous; steps on one context must
 * not overlap on different streams (they share workspaces).
 * Default path: three launches -- a prologue (controller, embedding), one persistent cooperative
 * kernel for every active layer and the LM head, and a finish kernel (acceptance, compaction).
 * When a step's context KV outweighs half a layer's weights (long contexts), the persistent kernel
 * is launched once per span of GEMM phases between two attentions and each layer's attention
 * runs as its own kernel (2 + 2 x active layers + 1 launches).
 * A step that does not fit the persistent kernel's shared-memory plan (tss_persistent_plan) is
 * rejected with TSS_ERR_UNSUPPORTED_ARCH before anything is enqueued.  With the environment
 * variable TSS_PATH=multi at tss_create, one kernel per operation runs instead, a diagnostic path
 * (bf16 GEMM activations: within the logit tolerance at the tiny test shape only; 6 + 7 x active
 * layers launches). */
tss_status tss_verify(tss_ctx* ctx, const tss_verify_batch* batch, const tss_kv_cache* kv,
                      const tss_verify_result* result, void* stream);

/* The attention kernel of the last step enqueued on ctx (tss_verify, tss_verify_grouped's last
 * group, tss_verify_profiled):
 *   0  the separate split-KV attention kernel (warp-level MMA; blocks of up to 64 rows),
 *   1  the tcgen05 attention kernel: blocks of at most 16 rows and head_dim 128, the keys on the
 *      MMA's 128-row side, K/V tiles by TMA, scores and outputs in tensor memory (the default for
 *      such steps; the environment variable TSS_ATTN_TC=0 at tss_create turns it off),
 *   2  the separate kernel's variant for blocks of more than 64 rows,
 *   3  the attention inside the persistent verify kernel;
 * -1 before the first step or for a NULL ctx.  Host state only: no CUDA call. */
int tss_attention_kernel(const tss_ctx* ctx);

/* Domain-grouped verification (a latency option for mixed-domain batches): the requests of the
 * batch are grouped by their skip set S(x) = Phi(d(x)) (Sec. "Domain-to-Configuration Mapping":
 * one model serves several domain-specific sparse paths), and one verification step per group is
 * enqueued on `stream`, the group with the fewest active layers first.  Each group's step streams
 * the weights of its own active layers only, so the requests of a domain that skips many layers
 * complete sooner than in the mixed step -- which streams the union of every request's active
 * layers once -- while the batch as a whole takes longer (the groups' layer counts add up to at
 * least the union).  Results land in the caller's arrays at each request's position, and every
 * request draws the same Philox uniforms as in tss_verify (counter request index = its index in
 * the whole batch), so the outputs equal tss_verify's up to the rounding of the GEMM partition.
 *   batch, kv, result: as tss_verify, DEVICE arrays only (io_host = 0).
 *   n_groups (optional, HOST): the number of groups (steps) enqueued.
 *   group_events (optional, HOST array of cudaEvent_t passed as void*, one per request, entries
 *   may be NULL): event g is recorded on `stream` when group g's results are in place, so a caller
 *   can time or wait for each group.
 * Uses the context's staging buffers: do not overlap with another call on the same context.
 * Errors: those of tss_verify (all checked for the whole batch before anything is enqueued);
 * INVALID_ARG for io_host != 0 or a uniform_stride above 512. */
tss_status tss_verify_grouped(tss_ctx* ctx, const tss_verify_batch* batch, const tss_kv_cache* kv,
                              const tss_verify_result* result, void* stream, int* n_groups,
                              void* const* group_events);

/* Prefill: append tokens to the requests' KV caches under their skip configurations (the
 * configuration is fixed for a whole request, prompt included: Sec. "Problem Formulation").
 * Request b's tokens [ctx_len[b], ctx_len[b] + n_tokens[b]) run through the layers its domain
 * does not skip, and their K/V rows are written to the cache of every such layer; layers it skips
 * are not touched.  Afterwards the caller's cache of request b holds ctx_len[b] + n_tokens[b]
 * tokens.  With head_dim 128 the requests of one skip set share passes of up to 4096 rows (each
 * request's next chunk at a multiple of 128 rows), every layer's projections run as tokens-tiled
 * tcgen05 GEMMs and its attention as a causal tcgen05 kernel (the environment variable
 * TSS_PREFILL=steps at tss_create selects the other path); otherwise the prompt runs in chains of
 * up to max_nodes tokens, each chain one verification step on the same kernels, whose acceptance
 * outputs are discarded.  The first call on the tcgen05 path allocates its workspaces (about
 * 0.45 GB at d_model 4096).
 *   n_tokens, ctx_len, domain_id, kv_slot: HOST arrays of n_req entries (n_tokens[b] >= 0;
 *     kv_slot NULL means slot b).
 *   tokens: the requests' tokens concatenated (sum(n_tokens) int32), DEVICE memory, or HOST
 *     memory when io_host != 0.
 * Asynchronous on `stream`, like tss_verify; host-detectable errors return before any launch. */
tss_status tss_prefill(tss_ctx* ctx, int n_req, const int32_t* n_tokens, const int32_t* ctx_len,
                       const int32_t* domain_id, const int32_t* kv_slot, const int32_t* tokens, int io_host,
                       const tss_kv_cache* kv, void* stream);

/* Synchronise `stream`, then return and clear the device status word (TSS_OK if no device-side
 * check failed since the last call). */
tss_status tss_sync_status(tss_ctx* ctx, void* stream);

/* Fault injection for tests of the device-side timeout path; no GPU fault is involved.  The next
 * n_steps verification steps of ctx on the persistent path do not publish one dataflow flag (the
 * first 128-feature tile of the residual after the first active layer), so the waits that need
 * it run out after the context's wait limit (environment variable TSS_WAIT_LIMIT_MS at
 * tss_create, 1..600000, default 2000 ms): the kernel records TSS_ERR_TIMEOUT in the status word,
 * every CTA leaves its loops and frees its tensor memory, and tss_sync_status reports the code.
 * That step's outputs are undefined.  The context stays usable: every step starts with fresh
 * counters and a clear abort word, so the next step runs normally.  A step with no active layer
 * withholds nothing.  n_steps = 0 cancels.  When the step's attention runs in the tcgen05 kernel
 * (tss_attention_kernel = 1), the first CTA of the step's first attention launch issues no MMA
 * instead, so that kernel's waits run out (after its fixed 2 s bound) and it takes the same
 * abort path; the next step's prologue resets its counters.  A tss_prefill call on the tcgen05
 * path also counts as a step: the first CTA of its first GEMM launch issues no MMA (2 s bound);
 * that call's cache rows are undefined. */
tss_status tss_inject_timeout(tss_ctx* ctx, int n_steps);

/* Diagnostic: the Philox4x32-10 stream that speculative sampling draws from when the batch gives
 * no uniforms, for one (seed, offset): counter (slot, request, offset lo, offset hi), key
 * (seed lo, seed hi), for requests [0, n_req) and slots [0, n_slots).
 *   words: DEVICE uint32 [n_req][n_slots][4] (16-byte aligned), the generator's four output words;
 *   uniforms: DEVICE fp32 [n_req][n_slots], (first word >> 8) * 2^-24, the value the acceptance
 *   uses.  Either may be NULL (not both).  n_req * n_slots <= 2^28.  Asynchronous on `stream`;
 *   uses the same device function as the acceptance kernels. */
tss_status tss_philox_uniforms(uint64_t seed, uint64_t offset, int n_req, int n_slots, uint32_t* words,
                               float* uniforms, void* stream);

/* Release everything the context owns (after the caller's streams are idle). NULL is a no-op. */
void tss_destroy(tss_ctx* ctx);

/* Plain bf16 weight-streaming linear layer on the library's GEMM kernel:
 *   y[m][o] = sum_k x[m][k] * w[o][k], x [m_rows][k_dim] bf16, w [n_out][k_dim] bf16,
 *   y [m_rows][n_out] fp32, all device, row-major; m_rows in [1, 256]; k_dim a multiple of 64;
 *   n_out a multiple of 128; rows of x and w 16-byte aligned.  The projections inside f_l
 *   (App. "Models") run on this kernel.  Uses the context's workspaces: do not overlap with a
 *   tss_verify of the same context. */
tss_status tss_linear(tss_ctx* ctx, const void* x, const void* w, float* y, int m_rows, int k_dim,
                      int n_out, void* stream);

/* Per-kernel device times of one verification step, by kernel kind:
 *   0 controller + embedding (+ RMSNorms on the multi-kernel path), 1 QKV GEMM (+RoPE, KV
 *   append), 2 attention, 3 O-projection GEMM, 4 gate/up GEMM (+SwiGLU), 5 down GEMM, 6 LM head
 *   GEMM (+argmax), 7 acceptance + KV compaction, 8 the persistent verify kernel (every active
 *   layer and the LM head in one launch; kinds 1-6 are then empty). */
#define TSS_KERNEL_KINDS 9
typedef struct {
  float ms[TSS_KERNEL_KINDS];     /* summed device time of the kind's launches */
  int launches[TSS_KERNEL_KINDS]; /* launches of the kind */
} tss_kernel_times;

/* Diagnostic twin of tss_verify: the same kernels without programmatic overlap, each bracketed by
 * a CUDA event pair, captured into a one-off graph and launched on `stream` (so the events time
 * device work only); synchronises the stream and ADDS the step's per-kind times into *times.
 * Results are written as by tss_verify. */
tss_status tss_verify_profiled(tss_ctx* ctx, const tss_verify_batch* batch, const tss_kv_cache* kv,
                               const tss_verify_result* result, void* stream, tss_kernel_times* times);

/* Allocation-free twin of tss_linear.  The paper has no counterpart: this entry point exists for
 * callers that cannot allocate device memory when they run the layer -- a plugin inside a host
 * framework that owns the whole device memory pool, a process with a memory budget fixed at
 * start-up, or a latency-critical loop that must not call cudaMalloc/cudaFree (they can
 * synchronise the device and stall unrelated streams).  It needs no tss_ctx and allocates
 * nothing: the stream-K scratch (partial tiles, per-tile counters) and a status word are
 * file-scope device arrays of the library, 8 MiB + 2 KiB in all.
 *   y[m][o] = sum_k x[m][k] * w[o][k]; x [m_rows][k_dim] bf16, w [n_out][k_dim] bf16,
 *   y [m_rows][n_out] fp32, device, row-major, 16-byte aligned; m_rows in [1, 64]; k_dim a
 *   multiple of 64; n_out a multiple of 128, at most 32768; and the scratch a problem needs,
 *   (min(#SMs, n_out/128 * k_dim/64) + n_out/128) * 128 * pad16(m_rows) * 4 bytes, at most 8 MiB
 *   -- larger requests return TSS_ERR_INVALID_ARG with a message.  The scratch bound caps n_out
 *   further for many rows: on a 152-SM GB300 with 49..64 rows, n_out <= (256 - 152) * 128 = 13312;
 *   with up to 16 rows the 32768 limit applies.
 * The arrays live in a CUDA module that the runtime loads on a device at the first call there
 * (CUDA's default lazy module loading), so the first call per device and process reserves the
 * 8 MiB; a caller that later gives the rest of the device memory to its own pool should make that
 * first call before, and before any stream capture (it also looks up the arrays' device addresses
 * and sets the kernel's shared-memory limit).  Later calls allocate and reserve nothing.  Every
 * call on a device shares the one array and the next call overwrites it (the counters are cleared
 * on `stream` at each call): calls that overlap on the GPU race, so serialise them on one stream.
 * Asynchronous on `stream`.  A device-side failure (a bounded wait that ran out) is recorded in
 * the status word that tss_linear_static_status reports; the result is then undefined. */
tss_status tss_linear_static(const void* x, const void* w, float* y, int m_rows, int k_dim, int n_out, void* stream);

/* Synchronise `stream`, then return and clear the status word of tss_linear_static on the current
 * device: TSS_OK, or TSS_ERR_TIMEOUT if a call since the last query gave up on a bounded wait
 * (its y is then undefined).  Allocates nothing. */
tss_status tss_linear_static_status(void* stream);

/* Diagnostic timeline of the last persistent-path step, recorded when the environment variable
 * TSS_TRACE=1 was set at tss_create: globaltimer nanoseconds, per CTA (row of
 * n_out / #SMs values), per phase pi (QKV, O, gate/up, down of each active layer in order, then
 * the LM head) at [pi*8 + 2*role + {0 first, 1 last}] for roles 0 weight TMA, 1 B operand,
 * 2 MMA, 3 epilogue, and the attention of layer slot j at [(4*64+1)*8 + 2j + {0,1}]; further
 * diagnostic slots follow (epilogue sub-steps of each phase's last segment, attention sub-steps
 * of layer slot 1).  0 = no activity.  With host == NULL only *n_out (values per device) is
 * returned.  Synchronises the device. */
tss_status tss_read_trace(tss_ctx* ctx, unsigned long long* host, size_t capacity, size_t* n_out);

const char* tss_status_string(tss_status s);
/* Message of the last error reported to the calling thread ("" if none). */
const char* tss_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* TSS_H */
