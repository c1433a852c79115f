// Host-visible launch interfaces shared by the library's translation units.
#pragma once

#include <string>
#include <utility>

#include "common.cuh"

namespace tss {

// Fused epilogues of the weight-streaming GEMM.
enum Epi : int {
  kEpiStore = 0,   // y[row][o] = acc (fp32), plain linear layer
  kEpiQkv = 1,     // RoPE on q/k, q -> bf16 buffer, k/v -> bf16 KV cache rows (KV append)
  kEpiResid = 2,   // h[row][o] += acc (O projection, down projection)
  kEpiSwiglu = 3,  // act[row][f] = bf16(silu(gate) * up) for interleaved gate/up tiles
  kEpiLmHead = 4,  // logits[row][v] (fp32, optional) + per-tile argmax partials
};

struct GemmParams {
  int n_tiles;      // output tiles of 128 weight rows
  int kb;           // k-blocks of 64 per tile
  int n_pad;        // MMA N = token rows padded to a multiple of 16 (<= 256)
  int stages;       // smem pipeline depth
  int n_acc_bufs;   // TMEM accumulator buffers (1 or 2)
  int slot;         // plan slot whose compacted rows feed the GEMM; -1: plain rows [0, m_raw)
  int m_raw;
  int layer_fixed;  // >= 0: TMA layer coordinate; -1: plan->act_layer[slot]
  const __nv_bfloat16* w_tiled;  // pre-tiled weights (bulk copies); nullptr: tensor-map TMA
  long long w_layer_elems;       // elements per layer in w_tiled
  const PlanDev* plan;
  const StepDesc* step;
  float* partials;  // stream-K partial tiles [(grid + n_tiles) * 128 * n_pad]
  int* counters;    // per-tile arrival counters (self-resetting)
  int* status;
  float* out;       // kEpiStore
  int out_ld;
  int o_real;
  float* h;         // kEpiResid: residual [kMaxRows][d_model]
  __nv_bfloat16* q_out;    // kEpiQkv: [kMaxRows][d_model]
  __nv_bfloat16* act_out;  // kEpiSwiglu: [kMaxRows][act_ld]
  int act_ld;
  const float* rope_cos;   // [max_positions][head_dim / 2]
  const float* rope_sin;
  float* amax_val;  // kEpiLmHead: [n_tiles][kMaxRows]
  int* amax_idx;
  int d_model, n_heads, head_dim, vocab;
};

size_t gemm_smem_bytes(int n_pad, int stages);
// TMEM columns for n_acc_bufs accumulators of n_pad fp32 columns (a power of two >= 32).
__host__ __device__ inline uint32_t gemm_tmem_cols(int n_pad, int n_acc_bufs) {
  uint32_t need = static_cast<uint32_t>(n_pad * n_acc_bufs);
  uint32_t c = 32;
  while (c < need) c <<= 1;
  return c;
}
cudaError_t gemm_prepare(size_t max_smem);
cudaError_t launch_gemm(int epi, const CUtensorMap& tmW, const CUtensorMap& tmX, const GemmParams& p, int grid,
                        size_t smem, cudaStream_t s, bool pdl);

struct AttnParams {
  int slot, n_splits, n_heads, d_model, head_dim;
  float scale_log2;  // log2(e) / sqrt(head_dim)
  const PlanDev* plan;
  const StepDesc* step;
  const __nv_bfloat16* q;  // [kMaxRows][d_model] compacted rows of the slot
  __nv_bfloat16* o;        // [kMaxRows][d_model]
  float* part_o;           // [B][H][n_splits][64 or 128][head_dim]
  float* part_ml;          // [B][H][n_splits][64 or 128][2]
  int wide;                // separate kernel: blocks of up to 128 rows (partials strided by 128, else 64)
  int* counters;           // [B][H], self-resetting
  int* status;
  XsLayout o_xs;           // o_xs.rows == 0: o row-major [row][d]; else split k-block tiled
};
size_t attn_smem_bytes(int head_dim);

// The tcgen05 attention for blocks of at most 16 rows and head_dim 128 (attn_tc.cu): one CTA per
// SM over the items' 128-key tiles laid end to end.
constexpr int kTcMaxNodes = 16;
constexpr int kTcMaxKeyTile = 128;
struct AttnTcParams {
  int slot, n_heads, d_model;
  float scale_log2;              // log2(e) / sqrt(head_dim)
  const PlanDev* plan;
  const StepDesc* step;
  const CUtensorMap* kv_maps;    // [n_layers] in device memory: each layer's cache as a 2-D bf16
                                 // tensor [n_slots * 2 * n_heads * cap rows][128], boxes 64 x 128, 128-byte swizzle
  const __nv_bfloat16* q;        // [kMaxRows][d_model] compacted rows (fp16 bits when o_xs.rows != 0)
  __nv_bfloat16* o;              // [kMaxRows][d_model], or the split tiled operand o_xs
  XsLayout o_xs;
  float* part_o;                 // [attn_tc_partial_rows][128]
  float* part_ml;                // [attn_tc_partial_rows][2]
  int* counters;                 // [B][H], self-resetting
  int* status;
  int withhold;                  // fault injection: CTA 0 issues no MMA (its first wait runs out)
};
// Compute-bound prefill (prefill.cu; head_dim 128): one pass = T rows holding the prompt chunks
// of requests with the same skip set, each chunk starting at a multiple of 128 rows (rows in the
// gaps have position -1 and write nothing).
constexpr int kPfEpiQkv = 0, kPfEpiResid = 1, kPfEpiSwiglu = 2;
struct PfParams {
  int T, n_qtiles, d_model, n_heads, head_dim, vocab, kv_cap;
  const int* row_pos;              // [T] position of each row's token, -1 for a gap row
  const int* row_slot;             // [T] KV slot of each row's request
  const int4* qtiles;              // [n_qtiles] (first row, slot, position of the first row, rows of the
                                   // request in the tile), heaviest first: the attention's work items
  float rms_eps;
  const int* tokens;               // [T] device
  const __nv_bfloat16* embed;      // [vocab][d]
  float* h;                        // [T_max][d] residual stream
  __nv_bfloat16 *xh, *xl;          // [T_max][x_ld] normed activations (hi, lo): the B operand of QKV and gate/up
  int x_ld;
  __nv_bfloat16 *qh, *ql;          // [T_max][d] q after RoPE (hi, lo)
  __nv_bfloat16 *ah, *al;          // [T_max][d] attention output (hi, lo): the B operand of O
  __nv_bfloat16 *uh, *ul;          // [T_max][u_ld] SwiGLU output (hi, lo): the B operand of down
  int u_ld;
  __nv_bfloat16* kv;               // this layer's cache [n_slots][2][H][cap][D]
  const float* rope_cos;           // [max_positions][D / 2]
  const float* rope_sin;
  int* status;
};
struct PfGemm {
  const __nv_bfloat16* w;          // pre-tiled weights (16 KiB blocks [layer][row tile][k-block])
  long long w_layer_elems;
  int layer, n_o, kb;              // layer, 128-row weight tiles, 64-column k-blocks
  int withhold;                    // fault injection: CTA 0 issues no MMA (its waits run out)
};
cudaError_t pf_prepare();
cudaError_t launch_pf_embed(const PfParams& p, cudaStream_t s);
cudaError_t launch_pf_norm(const PfParams& p, const float* g, cudaStream_t s);
cudaError_t launch_pf_gemm(int epi, const CUtensorMap& xh, const CUtensorMap& xl, const PfParams& p, const PfGemm& g,
                           int grid, cudaStream_t s);
cudaError_t launch_pf_attn(const CUtensorMap& qh, const CUtensorMap& ql, const CUtensorMap& kv, const PfParams& p,
                           cudaStream_t s);

size_t attn_tc_smem_bytes();
size_t attn_tc_partial_rows(int max_batch, int n_heads, int grid);
cudaError_t attn_tc_prepare();
cudaError_t launch_attention_tc(const AttnTcParams& p, int grid, cudaStream_t s, bool pdl);
cudaError_t attn_prepare();
cudaError_t launch_attention(const AttnParams& p, int B, cudaStream_t s, bool pdl);

struct MiscParams {
  const StepDesc* step;
  PlanDev* plan;
  int n_layers, d_model, n_heads, head_dim, vocab;
  float rms_eps;
  const __nv_bfloat16* embed;   // [vocab][d]
  float* h;                     // [kMaxRows][d]
  __nv_bfloat16* xn;            // [kMaxRows][d]
  const float* g_attn;          // [L][d]
  const float* g_mlp;           // [L][d]
  const float* g_final;         // [d]
  const float* amax_val;        // [n_vtiles][kMaxRows]
  const int* amax_idx;
  int n_vtiles;
  int* status;
  XsLayout xs;  // xs.rows == 0: xn row-major; else the persistent kernel's split tiled operand
};

cudaError_t misc_prepare();
cudaError_t launch_prologue(const MiscParams& p, float* ssp, int* zero_ints, int n_zero, int M, cudaStream_t s, bool pdl);
cudaError_t launch_finish(const MiscParams& p, int B, bool sample, cudaStream_t s, bool pdl);
// Dynamic shared memory of the sampling acceptance's staged inverse CDF: the vocabulary's weights
// with one skew word per 32 (0 when that exceeds kCdfStageMaxBytes: the unstaged pass runs).
constexpr size_t kCdfStageMaxBytes = 200 * 1024;
__host__ __device__ inline size_t cdf_stage_bytes(int vocab) {
  const size_t n = (static_cast<size_t>(vocab) + vocab / 32 + 1) * sizeof(float);
  return n <= kCdfStageMaxBytes ? n : 0;
}
cudaError_t launch_controller(const MiscParams& p, cudaStream_t s, bool pdl);
cudaError_t launch_embed(const MiscParams& p, int M, cudaStream_t s, bool pdl);
// which: 0 = attention norm of the slot's layer, 1 = MLP norm, 2 = final norm (slot ignored)
cudaError_t launch_rmsnorm(const MiscParams& p, int slot, int which, int M, cudaStream_t s, bool pdl);
cudaError_t launch_accept_greedy(const MiscParams& p, int B, cudaStream_t s, bool pdl);
cudaError_t launch_accept_sample(const MiscParams& p, int B, cudaStream_t s, bool pdl);
cudaError_t launch_compact(const MiscParams& p, int B, int n_act, cudaStream_t s, bool pdl);
cudaError_t launch_bf16_to_f32(const __nv_bfloat16* src, float* dst, size_t n, cudaStream_t s);
// The acceptance's Philox4x32-10 stream for one (seed, offset): words [n_req][n_slots][4] and/or
// uniforms [n_req][n_slots] (either may be null).
cudaError_t launch_philox_fill(uint64_t seed, uint64_t offset, int n_req, int n_slots, uint32_t* words, float* unif,
                               cudaStream_t s);
// Row-major [rows][cols] bf16 (rows % 128 == 0, cols % 64 == 0) -> pre-tiled, pre-swizzled blocks.
cudaError_t launch_tile_weights(const __nv_bfloat16* src, __nv_bfloat16* dst, int rows, int cols, cudaStream_t s);

// Persistent verify kernel (verify_mk.cu).
struct MkParams {
  int n_act, d, H, D, F_pad, Ft, V, V_pad, n_pad, stages, attn_splits, B, max_tiles;
  int kps;  // k-blocks (16 KiB of weights each) per pipeline stage
  XsLayout xs;  // B-operand layout (n_pad == xs.rows)
  int attn_plo;         // attention P.V with P split into hi/lo bf16 parts
  int w_evict_first;  // stream weights with the evict-first L2 policy
  int attn_extra;  // shared memory behind the ring that only the attention uses (bytes)
  // Phases [ph_begin, ph_end) run in this launch.  attn_external: the attention of each layer is a
  // separate kernel launched between the launches (long contexts), so none runs in here and an
  // O phase needs no flag from it.
  int ph_begin, ph_end, attn_external;
  unsigned long long* trace;  // optional timeline [grid][mk_trace_slots()], nullptr when off
  float eps, scale_log2;
  unsigned long long seq_base;  // epoch * 1024: flag values grow over steps, never reset
  const StepDesc* step;
  const PlanDev* plan;
  const __nv_bfloat16* w_qkv;  // pre-tiled weights [L][tiles][k-blocks][16 KiB]
  const __nv_bfloat16* w_o;
  const __nv_bfloat16* w_gu;
  const __nv_bfloat16* w_down;
  const __nv_bfloat16* w_lm;
  float* h;
  __nv_bfloat16* qbuf;
  __nv_bfloat16* obuf;
  __nv_bfloat16* act;
  __nv_bfloat16* xn;  // [kMaxRows][d] bf16(h * g) of the next norm phase, compacted rows
  float* partials0;  // stream-K partial tiles, alternating between consecutive phases
  float* partials1;
  int* counters;     // [7 kinds][max_tiles]
  float* ssp;        // [d/128][kMaxRows] per-tile partial sums of squares of h
  unsigned long long* hflag;    // [d/128]
  unsigned long long* qkvflag;  // [3d/128]
  unsigned long long* attflag;  // [max_batch][H]
  unsigned long long* guflag;   // [Ft]
  float* amax_val;
  int* amax_idx;
  float* attn_po;
  float* attn_pml;
  int* attn_cnt;
  const float* g_attn;
  const float* g_mlp;
  const float* g_final;
  const float* rope_cos;
  const float* rope_sin;
  int* status;
  int* abort_word;
  unsigned long long wait_ns;  // bound of every wait of the kernel
  int withhold_flag;  // fault injection: withhold one dataflow flag so that a bounded wait runs out
  int dp_tail;     // phases with a tile per CTA end with one whole tile per CTA (no fix-up on their tail)
};
size_t mk_smem_bytes(int n_pad, int parts, int stages, int head_dim, int kps, size_t attn_extra);
size_t mk_trace_slots();
cudaError_t mk_prepare();
int mk_max_blocks_per_sm(int head_dim, size_t smem);
cudaError_t launch_verify_mk(const MkParams& p, int grid, size_t smem, cudaStream_t s);

// Records the message tss_last_error() returns on the calling thread.
void set_last_error(const std::string& msg);

// Launch with optional programmatic dependent launch (the kernel may start while the previous
// kernel in the stream finishes; it calls griddepcontrol.wait before touching its outputs).
template <typename... KArgs, typename... Args>
cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s, bool pdl,
                     Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

}  // namespace tss
