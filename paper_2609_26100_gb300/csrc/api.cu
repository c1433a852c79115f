// C ABI and host runtime of the TSS verification library: weight repacking, workspace
// management, host-side validation, the per-step launch plan over the union of active layers,
// and CUDA-graph capture of that plan.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <string>
#include <tuple>
#include <vector>

#include "internal.h"

using namespace tss;

namespace {

thread_local std::string g_err;

tss_status fail(tss_status s, const std::string& msg) {
  g_err = msg;
  return s;
}

#define TSS_CU(call)                                                                           \
  do {                                                                                         \
    cudaError_t e_ = (call);                                                                   \
    if (e_ != cudaSuccess) return fail(TSS_ERR_CUDA, std::string(#call) + ": " + cudaGetErrorString(e_)); \
  } while (0)

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  if (!fn) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

// bf16 tensor [d2][d1][d0] (d0 innermost), box (64, rows, 1), 128-byte swizzle.  Weights use
// rank 3 (d2 = layer, loaded with 3-D TMA); activations use rank 2.
bool make_tmap(CUtensorMap* m, const void* base, uint64_t d0, uint64_t d1, uint64_t d2, uint32_t box_rows,
               int rank = 3) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {d0, d1, d2};
  cuuint64_t strides[2] = {d0 * 2, d0 * d1 * 2};
  cuuint32_t box[3] = {64, box_rows, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, static_cast<cuuint32_t>(rank), const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

int pad_to(int x, int m) { return (x + m - 1) / m * m; }

struct GraphKey {
  int B, M, n_act, mode, splits, attn;  // attn: the attention kernel variant (attn_variant)
  bool operator<(const GraphKey& o) const {
    return std::tie(B, M, n_act, mode, splits, attn) < std::tie(o.B, o.M, o.n_act, o.mode, o.splits, o.attn);
  }
};

constexpr int kRing = 4;
constexpr int kMaxPathStride = 1024;

}  // namespace

void tss::set_last_error(const std::string& msg) { g_err = msg; }

struct tss_ctx {
  tss_arch a{};
  int dev = 0, num_sms = 0;
  int L = 0, d = 0, H = 0, D = 0, F = 0, V = 0;
  int F_pad = 0, Ft = 0, V_pad = 0;
  // repacked weights
  __nv_bfloat16 *wqkv = nullptr, *wo = nullptr, *wgu = nullptr, *wdown = nullptr, *embed = nullptr, *lm = nullptr;
  float *g_attn = nullptr, *g_mlp = nullptr, *g_final = nullptr;
  float *rope_cos = nullptr, *rope_sin = nullptr;
  // workspaces
  float* h = nullptr;
  __nv_bfloat16 *xn = nullptr, *qbuf = nullptr, *obuf = nullptr, *act = nullptr;
  float* logits_ws = nullptr;
  float* partials = nullptr;
  size_t partials_floats = 0;
  int* counters = nullptr;
  float* amax_val = nullptr;
  int* amax_idx = nullptr;
  float *attn_po = nullptr, *attn_pml = nullptr;
  int* attn_cnt = nullptr;
  int max_splits = kMaxSplits;
  StepDesc* d_step = nullptr;
  StepDesc* h_ring[kRing] = {};
  cudaEvent_t ring_ev[kRing] = {};
  bool ring_used[kRing] = {};
  int ring_i = 0;
  PlanDev* d_plan = nullptr;
  std::vector<unsigned long long> phi;
  std::vector<int> phi_valid;
  int* d_status = nullptr;
  int* h_status = nullptr;
  // staging for host-pointer I/O
  int* io_tokens = nullptr;
  float* io_probs = nullptr;
  float* io_unif = nullptr;
  int* io_res = nullptr;  // accept[kMaxBatch] bonus[kMaxBatch] new_ctx[kMaxBatch] path[kMaxBatch*kMaxPathStride]
  // tensor maps
  std::map<int, CUtensorMap> tm_xn, tm_o, tm_act;
  // graphs
  std::map<GraphKey, cudaGraphExec_t> graphs;
  cudaStream_t cap_stream = nullptr;
  bool use_graphs = true;
  int gemm_ctas_per_sm = 2;
  // persistent verify kernel
  bool use_mk = true;
  int mk_kps = 3;  // weight k-blocks per ring stage of the persistent kernel (48 KiB stages measured best)
  int attn_mode = 0;  // 0 auto, 1 attention inside the persistent kernel, 2 separate attention kernels
  int w_evict_first = 1;
  int mk_max_stages = 12;
  int mk_dp_tail = 1;  // whole-tile tails for phases with a tile per CTA (TSS_MK_DP)
  int attn_plo = 1;
  int attn_splits_force = 0;  // > 0: key splits of the separate attention kernel (TSS_ATTN_SPLITS)
  int mk_splits_force = 0;    // > 0: key splits of the persistent kernel's attention (TSS_MK_ATTN_SPLITS)
  // tcgen05 attention of blocks of at most 16 rows (head_dim 128; TSS_ATTN_TC=0 turns it off)
  int attn_tc = 1;
  int last_attn = -1;                    // attention kernel of the last step (tss_attention_kernel)
  CUtensorMap* d_kvmaps = nullptr;       // [L] each layer's KV cache as a 2-D tensor
  std::vector<CUtensorMap> h_kvmaps;     // host copy of the last maps uploaded
  std::vector<const void*> kvmap_ptr;    // the layer pointers they were made for
  int kvmap_slots = -1, kvmap_cap = -1;  // ... and the cache shape
  bool kvmap_ok = false;                 // the maps describe the current cache
  float *tc_po = nullptr, *tc_pml = nullptr;
  // compute-bound prefill (prefill.cu; head_dim 128, TSS_PREFILL=steps turns it off)
  bool pf_enabled = true;
  int pf_tmax = 0;  // tokens per chunk; 0 until the workspaces exist
  float* pf_h = nullptr;
  __nv_bfloat16 *pf_xh = nullptr, *pf_xl = nullptr, *pf_qh = nullptr, *pf_ql = nullptr, *pf_ah = nullptr,
                *pf_al = nullptr, *pf_uh = nullptr, *pf_ul = nullptr;
  int* pf_tok = nullptr;
  int *pf_pos = nullptr, *pf_slot = nullptr;
  int4* pf_qt = nullptr;
  CUtensorMap pf_tm_xh, pf_tm_xl, pf_tm_qh, pf_tm_ql, pf_tm_ah, pf_tm_al, pf_tm_uh, pf_tm_ul;
  unsigned long long* trace = nullptr;  // persistent-kernel timeline when TSS_TRACE is set
  unsigned long long wait_ns = 2000000000ull;  // bound of the persistent kernel's waits (TSS_WAIT_LIMIT_MS)
  int inject_timeouts = 0;  // steps left that withhold one dataflow flag (tss_inject_timeout)
  unsigned long long epoch = 0;
  float* ssp = nullptr;
  unsigned long long* flags = nullptr;  // hflag | qkvflag | guflag | attflag
  int* mk_zero = nullptr;               // counters [7][max_tiles] | abort word | attention counters
  int mk_max_tiles = 0, mk_n_zero = 0;
  float *mk_part0 = nullptr, *mk_part1 = nullptr;
  size_t mk_part_floats = 0;
  std::vector<void*> allocs;
  size_t allocated = 0;    // bytes allocated by alloc()
  size_t alloc_limit = 0;  // > 0: alloc() fails beyond this many bytes (TSS_ALLOC_LIMIT_BYTES)

  template <typename T>
  tss_status alloc(T** p, size_t count) {
    const size_t bytes = count * sizeof(T) + 16;
    if (alloc_limit != 0 && allocated + bytes > alloc_limit)
      return fail(TSS_ERR_OUT_OF_MEMORY, "allocating " + std::to_string(bytes) + " more bytes would exceed the limit of " +
                                             std::to_string(alloc_limit) + " (TSS_ALLOC_LIMIT_BYTES)");
    void* q = nullptr;
    if (cudaMalloc(&q, bytes) != cudaSuccess) {
      cudaGetLastError();
      return fail(TSS_ERR_OUT_OF_MEMORY, "cudaMalloc of " + std::to_string(count * sizeof(T)) + " bytes failed");
    }
    allocs.push_back(q);
    allocated += bytes;
    *p = static_cast<T*>(q);
    return TSS_OK;
  }
};

namespace {

#define TSS_TRY(expr)              \
  do {                             \
    tss_status s_ = (expr);        \
    if (s_ != TSS_OK) return s_;   \
  } while (0)

struct GemmShape {
  int epi, n_tiles, kb;
  const CUtensorMap* tmW;
  const CUtensorMap* tmX;
};

void gemm_config(const tss_ctx* c, int n_pad, int n_tiles, int kb, int* grid, int* stages, size_t* smem, int* bufs) {
  const int per_sm = n_pad <= 64 ? c->gemm_ctas_per_sm : 1;
  const size_t budget = per_sm >= 2 ? 110 * 1024 : 220 * 1024;
  int s = 2;
  while (s < 12 && gemm_smem_bytes(n_pad, s + 1) <= budget) ++s;
  *stages = s;
  *smem = gemm_smem_bytes(n_pad, s);
  *bufs = n_pad <= 128 ? 2 : 1;
  long long T = static_cast<long long>(n_tiles) * kb;
  long long g = static_cast<long long>(c->num_sms) * per_sm;
  *grid = static_cast<int>(g < T ? g : T);
}

tss_status get_xmap(tss_ctx* c, std::map<int, CUtensorMap>& cache, const void* buf, int k, int n_pad,
                    const CUtensorMap** out) {
  auto it = cache.find(n_pad);
  if (it == cache.end()) {
    CUtensorMap m;
    if (!make_tmap(&m, buf, static_cast<uint64_t>(k), kMaxRows, 1, static_cast<uint32_t>(n_pad), 2))
      return fail(TSS_ERR_CUDA, "cuTensorMapEncodeTiled failed for an activation buffer");
    it = cache.emplace(n_pad, m).first;
  }
  *out = &it->second;
  return TSS_OK;
}

MiscParams misc_params(tss_ctx* c) {
  MiscParams p{};
  p.step = c->d_step;
  p.plan = c->d_plan;
  p.n_layers = c->L;
  p.d_model = c->d;
  p.n_heads = c->H;
  p.head_dim = c->D;
  p.vocab = c->V;
  p.rms_eps = c->a.rms_eps;
  p.embed = c->embed;
  p.h = c->h;
  p.xn = c->xn;
  p.g_attn = c->g_attn;
  p.g_mlp = c->g_mlp;
  p.g_final = c->g_final;
  p.amax_val = c->amax_val;
  p.amax_idx = c->amax_idx;
  p.n_vtiles = c->V_pad / 128;
  p.status = c->d_status;
  return p;
}

GemmParams gemm_base(tss_ctx* c, int n_pad) {
  GemmParams g{};
  g.n_pad = n_pad;
  g.plan = c->d_plan;
  g.step = c->d_step;
  g.partials = c->partials;
  g.counters = c->counters;
  g.status = c->d_status;
  g.h = c->h;
  g.q_out = c->qbuf;
  g.act_out = c->act;
  g.act_ld = c->F_pad;
  g.rope_cos = c->rope_cos;
  g.rope_sin = c->rope_sin;
  g.amax_val = c->amax_val;
  g.amax_idx = c->amax_idx;
  g.d_model = c->d;
  g.n_heads = c->H;
  g.head_dim = c->D;
  g.vocab = c->V;
  g.layer_fixed = -1;
  return g;
}

tss_status run_gemm(tss_ctx* c, int epi, const CUtensorMap& tmW, const CUtensorMap& tmX, GemmParams g, int n_tiles,
                    int kb, cudaStream_t s, bool pdl) {
  int grid, stages, bufs;
  size_t smem;
  gemm_config(c, g.n_pad, n_tiles, kb, &grid, &stages, &smem, &bufs);
  g.n_tiles = n_tiles;
  g.kb = kb;
  g.stages = stages;
  g.n_acc_bufs = bufs;
  if (static_cast<size_t>(grid + n_tiles) * 128 * g.n_pad > c->partials_floats)
    return fail(TSS_ERR_INVALID_ARG, "GEMM partial workspace too small");
  TSS_CU(launch_gemm(epi, tmW, tmX, g, grid, smem, s, pdl));
  return TSS_OK;
}

struct StepPlan {
  int B, M, n_act, mode, splits, n_pad;
  int max_nodes;      // rows of the largest request's block
  int tiles;          // 64-key tiles of the longest request (context + block)
  long long ctx_sum;  // context tokens over the batch
};

// The attention kernel of a step: 2 the separate kernel's wide variant (blocks over 64 rows), 1
// the tcgen05 kernel (blocks of at most kTcMaxNodes rows, head_dim 128, KV tensor maps of the
// current cache uploaded), 0 the separate kernel's narrow variant.
int attn_variant(const tss_ctx* c, const StepPlan& sp) {
  if (sp.max_nodes > kNarrowNodes) return 2;
  if (c->attn_tc && c->D == 128 && sp.max_nodes <= kTcMaxNodes && c->kvmap_ok) return 1;
  return 0;
}

AttnTcParams tc_params(const tss_ctx* c, float scale_log2) {
  AttnTcParams tp{};
  tp.n_heads = c->H;
  tp.d_model = c->d;
  tp.scale_log2 = scale_log2;
  tp.plan = c->d_plan;
  tp.step = c->d_step;
  tp.kv_maps = c->d_kvmaps;
  tp.q = c->qbuf;
  tp.o = c->obuf;
  tp.part_o = c->tc_po;
  tp.part_ml = c->tc_pml;
  tp.counters = c->attn_cnt;
  tp.status = c->d_status;
  return tp;
}

// Tensor maps of the KV cache for the tcgen05 attention, one per layer: the layer's buffer as a
// 2-D bf16 tensor of n_slots * 2 * n_heads * cap rows of 128 elements.  Encoded and uploaded (in
// stream order, before the step's kernels) only when the cache's pointers or shape change, so a
// captured graph keeps reading the maps from the same device array.
tss_status sync_kv_maps(tss_ctx* c, const tss_kv_cache* kv, cudaStream_t s) {
  if (!c->attn_tc || !c->d_kvmaps) return TSS_OK;
  bool same = c->kvmap_slots == kv->n_slots && c->kvmap_cap == kv->cap;
  for (int l = 0; l < c->L && same; ++l) same = c->kvmap_ptr[l] == kv->layer[l];
  if (same) return TSS_OK;
  const unsigned long long rows = static_cast<unsigned long long>(kv->n_slots) * 2ull * c->H * kv->cap;
  c->kvmap_ok = false;
  c->kvmap_slots = kv->n_slots;
  c->kvmap_cap = kv->cap;
  for (int l = 0; l < c->L; ++l) c->kvmap_ptr[l] = kv->layer[l];
  if (rows == 0 || rows + kTcMaxKeyTile > 0x7fffffffull) return TSS_OK;  // (row coordinates are 32-bit)
  for (int l = 0; l < c->L; ++l) {
    std::memset(&c->h_kvmaps[l], 0, sizeof(CUtensorMap));
    if (kv->layer[l] && !make_tmap(&c->h_kvmaps[l], kv->layer[l], 128, rows, 1, 128, 2))
      return fail(TSS_ERR_CUDA, "cuTensorMapEncodeTiled failed for a KV cache layer");
  }
  TSS_CU(cudaMemcpyAsync(c->d_kvmaps, c->h_kvmaps.data(), sizeof(CUtensorMap) * c->L, cudaMemcpyHostToDevice, s));
  c->kvmap_ok = true;
  return TSS_OK;
}

// Optional per-launch event timing (tss_verify_profiled).
struct Prof {
  std::vector<cudaEvent_t> ev;
  std::vector<int> kind;
  cudaStream_t s = nullptr;
  bool capturing = false;  // under stream capture an event record must be an external node
  cudaError_t record(cudaEvent_t e) {
    return capturing ? cudaEventRecordWithFlags(e, s, cudaEventRecordExternal) : cudaEventRecord(e, s);
  }
  tss_status begin(int k) {
    cudaEvent_t e;
    TSS_CU(cudaEventCreate(&e));
    ev.push_back(e);
    kind.push_back(k);
    TSS_CU(record(e));
    return TSS_OK;
  }
  tss_status end() {
    cudaEvent_t e;
    TSS_CU(cudaEventCreate(&e));
    ev.push_back(e);
    kind.push_back(-1);
    TSS_CU(record(e));
    return TSS_OK;
  }
};

// Enqueue every kernel of one verification step (also used under stream capture).  With a Prof,
// every launch is bracketed by events and launched without programmatic overlap.
tss_status enqueue_step(tss_ctx* c, const StepPlan& sp, cudaStream_t s, Prof* prof = nullptr) {
  const bool pdl = prof == nullptr;
#define TSS_K(kind, expr)                       \
  do {                                          \
    if (prof) TSS_TRY(prof->begin(kind));       \
    expr;                                       \
    if (prof) TSS_TRY(prof->end());             \
  } while (0)
  MiscParams mp = misc_params(c);
  const int n_pad = sp.n_pad;
  const CUtensorMap *txn, *to, *tact;
  TSS_TRY(get_xmap(c, c->tm_xn, c->xn, c->d, n_pad, &txn));
  TSS_TRY(get_xmap(c, c->tm_o, c->obuf, c->d, n_pad, &to));
  TSS_TRY(get_xmap(c, c->tm_act, c->act, c->F_pad, n_pad, &tact));

  TSS_K(0, TSS_CU(launch_controller(mp, s, false)));
  TSS_K(0, TSS_CU(launch_embed(mp, sp.M, s, pdl)));
  AttnParams ap{};
  ap.n_splits = sp.splits;
  ap.n_heads = c->H;
  ap.d_model = c->d;
  ap.head_dim = c->D;
  ap.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(c->D)));
  ap.plan = c->d_plan;
  ap.step = c->d_step;
  ap.q = c->qbuf;
  ap.o = c->obuf;
  ap.part_o = c->attn_po;
  ap.part_ml = c->attn_pml;
  ap.wide = sp.max_nodes > kNarrowNodes ? 1 : 0;
  ap.counters = c->attn_cnt;
  ap.status = c->d_status;
  const bool tc = attn_variant(c, sp) == 1;
  AttnTcParams tp = tc_params(c, ap.scale_log2);
  const int kbd = c->d / 64;
  for (int j = 0; j < sp.n_act; ++j) {
    // attention sub-block: h_{l+1} = f_l(h_l) only for layers in the union; others get no launch
    TSS_K(0, TSS_CU(launch_rmsnorm(mp, j, 0, sp.M, s, pdl)));
    GemmParams g = gemm_base(c, n_pad);
    g.slot = j;
    const size_t dd = static_cast<size_t>(c->d) * c->d;
    g.w_tiled = c->wqkv;
    g.w_layer_elems = static_cast<long long>(3 * dd);
    TSS_K(1, TSS_TRY(run_gemm(c, kEpiQkv, *txn, *txn, g, 3 * c->d / 128, kbd, s, pdl)));
    if (tc) {
      tp.slot = j;
      TSS_K(2, TSS_CU(launch_attention_tc(tp, c->num_sms, s, pdl)));
    } else {
      ap.slot = j;
      TSS_K(2, TSS_CU(launch_attention(ap, sp.B, s, pdl)));
    }
    g.w_tiled = c->wo;
    g.w_layer_elems = static_cast<long long>(dd);
    TSS_K(3, TSS_TRY(run_gemm(c, kEpiResid, *to, *to, g, c->d / 128, kbd, s, pdl)));
    // feed-forward sub-block
    TSS_K(0, TSS_CU(launch_rmsnorm(mp, j, 1, sp.M, s, pdl)));
    g.w_tiled = c->wgu;
    g.w_layer_elems = static_cast<long long>(c->Ft) * 128 * c->d;
    TSS_K(4, TSS_TRY(run_gemm(c, kEpiSwiglu, *txn, *txn, g, c->Ft, kbd, s, pdl)));
    g.w_tiled = c->wdown;
    g.w_layer_elems = static_cast<long long>(c->d) * c->F_pad;
    TSS_K(5, TSS_TRY(run_gemm(c, kEpiResid, *tact, *tact, g, c->d / 128, c->F_pad / 64, s, pdl)));
  }
  TSS_K(0, TSS_CU(launch_rmsnorm(mp, kFinalSlot, 2, sp.M, s, pdl)));
  GemmParams g = gemm_base(c, n_pad);
  g.slot = kFinalSlot;
  g.layer_fixed = 0;
  g.w_tiled = c->lm;
  g.w_layer_elems = 0;
  TSS_K(6, TSS_TRY(run_gemm(c, kEpiLmHead, *txn, *txn, g, c->V_pad / 128, kbd, s, pdl)));
  if (sp.mode == TSS_MODE_SAMPLE) {
    TSS_K(7, TSS_CU(launch_accept_sample(mp, sp.B, s, pdl)));
  } else {
    TSS_K(7, TSS_CU(launch_accept_greedy(mp, sp.B, s, pdl)));
  }
  TSS_K(7, TSS_CU(launch_compact(mp, sp.B, sp.n_act, s, pdl)));
#undef TSS_K
  return TSS_OK;
}

// Shared-memory plan of the persistent kernel: the ring (stages x kps weight blocks with their
// B-operand blocks) and, behind it, attention-only space so that the attention, which borrows
// the ring, keeps all key tiles of a split resident (or as many as fit, in rounds).
struct MkConfig {
  int kps = 0, stages = 0, attn_splits = 1;
  size_t attn_extra = 0, smem = 0;
};

// Key splits per (request, head) for the persistent kernel's attention: the fewest waves of
// items over the grid times the tiles an item scores, plus a fixed per-item cost (flags, merge)
// of about three tiles.  Short contexts get about one item per CTA.
// What the persistent kernel's shared-memory plan depends on (a context's shape and switches).
struct MkPlanIn {
  int D, H, num_sms, kps_max, stages_max, max_splits;
  int splits_force;  // > 0: key splits of the persistent kernel's attention (TSS_MK_ATTN_SPLITS)
};
MkPlanIn mk_plan_in(const tss_ctx* c) {
  return MkPlanIn{c->D, c->H, c->num_sms, c->mk_kps, c->mk_max_stages, c->max_splits, c->mk_splits_force};
}

int mk_attn_splits(const MkPlanIn& c, int B, int tiles) {
  const int pairs = B * c.H;
  int best = 1;
  long long best_cost = -1;
  for (int sl = 1; sl <= c.max_splits; ++sl) {
    if (sl > 1 && sl > tiles) break;
    const long long waves = (static_cast<long long>(pairs) * sl + c.num_sms - 1) / c.num_sms;
    const long long cost = waves * ((tiles + sl - 1) / sl + 3);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = sl;
    }
  }
  return best;
}

// Key splits per (request, head) for the separate attention kernel (two CTAs per SM).  In units
// of one CTA scoring one 64-key tile, the launch takes about the larger of the mean load of a CTA
// slot and the longest item, and every item costs about kItemTiles more for its set-up and the
// merge of the splits.  The fewest splits on ties.  In a batch of ragged contexts this splits the
// long requests' items so that they no longer set the length of the launch (13B batch of
// contexts 644-3059: two splits, 98.6 vs 115.1 us per layer); equal long contexts keep one.
int ext_attn_splits(const tss_ctx* c, const StepDesc* sd, int B) {
  constexpr long long kItemTiles = 3;
  const long long slots = 2LL * c->num_sms;
  int max_tiles = 1;
  for (int b = 0; b < B; ++b) max_tiles = std::max(max_tiles, (sd->req_ctx[b] + sd->req_nodes[b] + 63) / 64);
  int best = 1;
  long long best_cost = -1;
  for (int sl = 1; sl <= c->max_splits && (sl == 1 || sl <= max_tiles); ++sl) {
    long long work = 0, longest = 0;
    for (int b = 0; b < B; ++b) {
      const long long t = (sd->req_ctx[b] + sd->req_nodes[b] + 63) / 64;
      const long long per = (t + sl - 1) / sl;
      const long long items = per > 0 ? (t + per - 1) / per : 0;
      work += c->H * (t + items * kItemTiles);
      longest = std::max(longest, per + kItemTiles);
    }
    const long long cost = std::max((work + slots - 1) / slots, longest);
    if (best_cost < 0 || cost < best_cost) {
      best_cost = cost;
      best = sl;
    }
  }
  return best;
}

// B requests with M rows in all, the longest one spanning `tiles` 64-key tiles.
bool mk_config_for(const MkPlanIn& c, int B, int M, int tiles, MkConfig* out) {
  constexpr size_t kLimit = 232448;  // per-block shared-memory maximum of sm_103 (227 KiB)
  const size_t q = static_cast<size_t>(kNarrowNodes) * (c.D + 8) * 2;
  const size_t tile = static_cast<size_t>(2) * 64 * (c.D + 8) * 2;
  const int splits = c.splits_force > 0 ? std::min(c.splits_force, c.max_splits) : mk_attn_splits(c, B, std::max(tiles, 1));
  const int per = std::max(1, (std::max(tiles, 1) + splits - 1) / splits);
  for (int kps = c.kps_max; kps >= 1; --kps) {
    const XsLayout xs = xs_layout(M);
    const size_t stage = static_cast<size_t>(kps) * (16384 + static_cast<size_t>(xs.rows) * xs.parts * 128);
    for (int S = c.stages_max; S >= 2; --S) {
      const size_t ring = S * stage;
      const size_t base = mk_smem_bytes(xs.rows, xs.parts, S, c.D, kps, 0);
      if (base > kLimit) continue;
      const size_t avail = kLimit - base;
      // at least Q + one tile, and Q + the warps' merge buffer (8 warps x 16 rows x D floats)
      const size_t first = q + std::max(tile, static_cast<size_t>(8) * 16 * c.D * 4);
      const size_t need_min = ring >= first ? 0 : first - ring;
      if (need_min > avail) continue;
      const size_t want = q + per * tile > ring ? q + per * tile - ring : 0;
      size_t extra = std::max(need_min, std::min(want, avail));
      extra = (extra + 15) & ~size_t(15);
      if (base + extra > kLimit) extra = need_min;
      out->kps = kps;
      out->stages = S;
      out->attn_splits = splits;
      out->attn_extra = extra;
      out->smem = base + extra;
      return true;
    }
  }
  return false;
}

bool mk_config(const tss_ctx* c, const StepPlan& sp, MkConfig* out) {
  return mk_config_for(mk_plan_in(c), sp.B, sp.M, sp.tiles, out);
}

// One verification step on the persistent path: prologue (controller, embedding, sums of
// squares), the persistent verify kernel (all layers + LM head), finish (acceptance + KV
// compaction).
tss_status enqueue_step_mk(tss_ctx* c, const StepPlan& sp, cudaStream_t s, Prof* prof) {
  MiscParams mp = misc_params(c);
  // the persistent kernel takes its B operands split into hi/lo parts in the k-block tiled layout
  const XsLayout xs = xs_layout(sp.M);
  const int n_pad = xs.rows;
  mp.xs = xs;
  MkConfig cfg;
  if (!mk_config(c, sp, &cfg)) return fail(TSS_ERR_UNSUPPORTED_ARCH, "persistent kernel: no shared-memory plan");
  const int kps = cfg.kps, stages = cfg.stages;
  const size_t smem = cfg.smem;
  const int nt = c->d / 128;
  MkParams p{};
  p.n_act = sp.n_act;
  p.d = c->d;
  p.H = c->H;
  p.D = c->D;
  p.F_pad = c->F_pad;
  p.Ft = c->Ft;
  p.V = c->V;
  p.V_pad = c->V_pad;
  p.n_pad = n_pad;
  p.stages = stages;
  p.kps = kps;
  p.xs = xs;
  p.dp_tail = c->mk_dp_tail;
  p.attn_plo = c->attn_plo;
  p.attn_extra = static_cast<int>(cfg.attn_extra);
  p.w_evict_first = c->w_evict_first;
  p.attn_splits = cfg.attn_splits;
  p.B = sp.B;
  p.max_tiles = c->mk_max_tiles;
  p.trace = c->trace;
  p.eps = c->a.rms_eps;
  p.scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(c->D)));
  p.seq_base = ++c->epoch * 1024ull;
  p.step = c->d_step;
  p.plan = c->d_plan;
  p.w_qkv = c->wqkv;
  p.w_o = c->wo;
  p.w_gu = c->wgu;
  p.w_down = c->wdown;
  p.w_lm = c->lm;
  p.h = c->h;
  p.qbuf = c->qbuf;
  p.obuf = c->obuf;
  p.act = c->act;
  p.xn = c->xn;
  p.partials0 = c->mk_part0;
  p.partials1 = c->mk_part1;
  p.counters = c->mk_zero;
  p.abort_word = c->mk_zero + 7 * c->mk_max_tiles;
  p.ssp = c->ssp;
  p.hflag = c->flags;
  p.qkvflag = c->flags + nt;
  p.guflag = c->flags + 4 * nt;
  p.attflag = c->flags + 4 * nt + c->Ft;
  p.amax_val = c->amax_val;
  p.amax_idx = c->amax_idx;
  p.attn_po = c->attn_po;
  p.attn_pml = c->attn_pml;
  p.attn_cnt = c->attn_cnt;
  p.g_attn = c->g_attn;
  p.g_mlp = c->g_mlp;
  p.g_final = c->g_final;
  p.rope_cos = c->rope_cos;
  p.rope_sin = c->rope_sin;
  p.status = c->d_status;
  p.wait_ns = c->wait_ns;
  p.withhold_flag = c->inject_timeouts > 0 && sp.n_act > 0 ? 1 : 0;
  if (p.withhold_flag) --c->inject_timeouts;
#define TSS_MK(kind, expr)                 \
  do {                                     \
    if (prof) TSS_TRY(prof->begin(kind));  \
    expr;                                  \
    if (prof) TSS_TRY(prof->end());        \
  } while (0)
  // Long contexts: the KV stream outweighs the weights, and the attention wants more warps per
  // SM than the persistent kernel has; each layer's attention is then a separate kernel between
  // launches of the persistent kernel over the GEMM phases in between.
  const double layer_bytes = (4.0 * c->d * c->d + 3.0 * c->d * c->a.d_mlp) * 2.0;
  const double kv_bytes = static_cast<double>(sp.ctx_sum) * 4.0 * c->d;
  // (blocks of more than 64 rows always take the separate kernels: their wide variant has the eight
  // query tiles and 128-row buffers; the attention inside the persistent kernel keeps 64)
  // Also when the (request, head) items outnumber the CTAs: inside the persistent kernel they
  // would run in more than one wave, one CTA per SM (13B, 4 requests x 40 heads, contexts ~2000:
  // 7.6 ms with separate kernels vs 11.2 ms inside).
  const bool ext = sp.max_nodes > kNarrowNodes || c->attn_mode == 2 ||
                   (c->attn_mode == 0 && (kv_bytes >= 0.5 * layer_bytes || sp.B * c->H > c->num_sms));
  p.attn_external = ext ? 1 : 0;
  c->last_attn = ext ? attn_variant(c, sp) : 3;
  TSS_MK(0, TSS_CU(launch_prologue(mp, c->ssp, c->mk_zero, c->mk_n_zero, sp.M, s, false)));
  if (!ext) {
    p.ph_begin = 0;
    p.ph_end = 1 << 30;
    TSS_MK(8, TSS_CU(launch_verify_mk(p, c->num_sms, smem, s)));
  } else {
    AttnParams ap{};
    ap.n_splits = sp.splits;
    ap.n_heads = c->H;
    ap.d_model = c->d;
    ap.head_dim = c->D;
    ap.scale_log2 = p.scale_log2;
    ap.plan = c->d_plan;
    ap.step = c->d_step;
    ap.q = c->qbuf;
    ap.o = c->obuf;
    ap.o_xs = xs;  // fp16 q, hi/lo output: the persistent kernel's operands
    ap.part_o = c->attn_po;
    ap.part_ml = c->attn_pml;
    ap.wide = sp.max_nodes > kNarrowNodes ? 1 : 0;
    ap.counters = c->attn_cnt;
    ap.status = c->d_status;
    const bool tc = attn_variant(c, sp) == 1;
    AttnTcParams tp = tc_params(c, p.scale_log2);
    tp.o_xs = xs;
    // fault injection: with the tcgen05 attention the first attention launch withholds the signal
    // (the persistent launches then withhold nothing)
    const int inject_attn = tc ? p.withhold_flag : 0;
    if (tc) p.withhold_flag = 0;
    int pb = 0;
    for (int j = 0; j < sp.n_act; ++j) {
      p.ph_begin = pb;  // phases 4j .. 4j+3 are QKV, O, gate/up, down of slot j; 4 n_act the LM head
      p.ph_end = 4 * j + 1;
      TSS_MK(8, TSS_CU(launch_verify_mk(p, c->num_sms, smem, s)));
      if (tc) {
        tp.slot = j;
        tp.withhold = j == 0 ? inject_attn : 0;
        TSS_MK(2, TSS_CU(launch_attention_tc(tp, c->num_sms, s, prof == nullptr)));
      } else {
        ap.slot = j;
        TSS_MK(2, TSS_CU(launch_attention(ap, sp.B, s, false)));
      }
      pb = 4 * j + 1;
    }
    p.ph_begin = pb;
    p.ph_end = 1 << 30;
    TSS_MK(8, TSS_CU(launch_verify_mk(p, c->num_sms, smem, s)));
  }
  TSS_MK(7, TSS_CU(launch_finish(mp, sp.B, sp.mode == TSS_MODE_SAMPLE, s, false)));
#undef TSS_MK
  return TSS_OK;
}

bool mk_supported(const tss_ctx* c, const StepPlan& sp) {
  if (!c->use_mk) return false;
  MkConfig cfg;
  if (!mk_config(c, sp, &cfg)) return false;
  return mk_max_blocks_per_sm(c->D, cfg.smem) >= 1;
}

tss_status validate_arch(const tss_arch* a) {
  if (!a) return fail(TSS_ERR_INVALID_ARG, "arch is NULL");
  if (a->n_layers < 1 || a->n_layers > kMaxLayers) return fail(TSS_ERR_UNSUPPORTED_ARCH, "n_layers must be in [1, 64]");
  if (a->head_dim != 64 && a->head_dim != 128) return fail(TSS_ERR_UNSUPPORTED_ARCH, "head_dim must be 64 or 128");
  if (a->n_heads < 1 || a->d_model != a->n_heads * a->head_dim)
    return fail(TSS_ERR_UNSUPPORTED_ARCH, "d_model must equal n_heads * head_dim");
  if (a->d_model % 128 != 0) return fail(TSS_ERR_UNSUPPORTED_ARCH, "d_model must be a multiple of 128");
  if (a->d_model > 8192) return fail(TSS_ERR_UNSUPPORTED_ARCH, "d_model must be at most 8192");
  if (a->d_mlp < 1 || a->vocab < 1) return fail(TSS_ERR_UNSUPPORTED_ARCH, "d_mlp and vocab must be positive");
  if (a->d_mlp % 8 != 0) return fail(TSS_ERR_UNSUPPORTED_ARCH, "d_mlp must be a multiple of 8");
  if (a->max_batch < 1 || a->max_batch > kMaxBatch) return fail(TSS_ERR_INVALID_ARG, "max_batch must be in [1, 64]");
  if (a->max_rows < 1 || a->max_rows > kMaxRows) return fail(TSS_ERR_INVALID_ARG, "max_rows must be in [1, 256]");
  if (a->max_nodes < 1 || a->max_nodes > kMaxNodes) return fail(TSS_ERR_INVALID_ARG, "max_nodes must be in [1, 128]");
  if (a->max_domains < 1 || a->max_domains > (1 << 20)) return fail(TSS_ERR_INVALID_ARG, "max_domains out of range");
  if (a->max_positions < 1) return fail(TSS_ERR_INVALID_ARG, "max_positions must be positive");
  if (!(a->rms_eps >= 0.f) || !(a->rope_theta > 0.f)) return fail(TSS_ERR_INVALID_ARG, "rms_eps / rope_theta invalid");
  return TSS_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

tss_status build_weights(tss_ctx* c, const tss_weights* w) {
  const int L = c->L, d = c->d, F = c->F, V = c->V;
  if (!w || !w->embed || !w->lm_head || !w->final_norm || !w->attn_norm || !w->wq || !w->wk || !w->wv || !w->wo ||
      !w->mlp_norm || !w->w_gate || !w->w_up || !w->w_down)
    return fail(TSS_ERR_INVALID_ARG, "a weight pointer is NULL");
  for (int l = 0; l < L; ++l)
    if (!w->attn_norm[l] || !w->wq[l] || !w->wk[l] || !w->wv[l] || !w->wo[l] || !w->mlp_norm[l] || !w->w_gate[l] ||
        !w->w_up[l] || !w->w_down[l])
      return fail(TSS_ERR_INVALID_ARG, "weights of layer " + std::to_string(l) + " incomplete");
  const size_t dd = static_cast<size_t>(d) * d;
  const size_t gu_rows = static_cast<size_t>(c->Ft) * 128;
  TSS_TRY(c->alloc(&c->wqkv, static_cast<size_t>(L) * 3 * dd));
  TSS_TRY(c->alloc(&c->wo, static_cast<size_t>(L) * dd));
  TSS_TRY(c->alloc(&c->wgu, static_cast<size_t>(L) * gu_rows * d));
  TSS_TRY(c->alloc(&c->wdown, static_cast<size_t>(L) * d * c->F_pad));
  TSS_TRY(c->alloc(&c->embed, static_cast<size_t>(V) * d));
  TSS_TRY(c->alloc(&c->lm, static_cast<size_t>(c->V_pad) * d));
  TSS_TRY(c->alloc(&c->g_attn, static_cast<size_t>(L) * d));
  TSS_TRY(c->alloc(&c->g_mlp, static_cast<size_t>(L) * d));
  TSS_TRY(c->alloc(&c->g_final, d));
  const size_t b2 = sizeof(__nv_bfloat16);
  // Row-major staging of one matrix at a time, then tiling into the library's pre-tiled layout.
  size_t tmp_elems = std::max(std::max(3 * dd, gu_rows * d), std::max(static_cast<size_t>(d) * c->F_pad,
                                                                        static_cast<size_t>(c->V_pad) * d));
  __nv_bfloat16* tmp = nullptr;
  if (cudaMalloc(&tmp, tmp_elems * b2) != cudaSuccess) {
    cudaGetLastError();
    return fail(TSS_ERR_OUT_OF_MEMORY, "weight staging allocation failed");
  }
  struct Free {
    void* p;
    ~Free() { cudaFree(p); }
  } free_tmp{tmp};
  TSS_CU(cudaMemcpy(c->embed, w->embed, static_cast<size_t>(V) * d * b2, cudaMemcpyDeviceToDevice));
  TSS_CU(cudaMemset(tmp, 0, static_cast<size_t>(c->V_pad) * d * b2));
  TSS_CU(cudaMemcpy(tmp, w->lm_head, static_cast<size_t>(V) * d * b2, cudaMemcpyDeviceToDevice));
  TSS_CU(launch_tile_weights(tmp, c->lm, c->V_pad, d, 0));
  TSS_CU(launch_bf16_to_f32(static_cast<const __nv_bfloat16*>(w->final_norm), c->g_final, d, 0));
  for (int l = 0; l < L; ++l) {
    TSS_CU(cudaMemcpy(tmp, w->wq[l], dd * b2, cudaMemcpyDeviceToDevice));
    TSS_CU(cudaMemcpy(tmp + dd, w->wk[l], dd * b2, cudaMemcpyDeviceToDevice));
    TSS_CU(cudaMemcpy(tmp + 2 * dd, w->wv[l], dd * b2, cudaMemcpyDeviceToDevice));
    TSS_CU(launch_tile_weights(tmp, c->wqkv + static_cast<size_t>(l) * 3 * dd, 3 * d, d, 0));
    TSS_CU(launch_tile_weights(static_cast<const __nv_bfloat16*>(w->wo[l]), c->wo + static_cast<size_t>(l) * dd, d, d, 0));
    // gate/up interleaved per 64 features: tile t = [gate rows 64t..64t+63 ; up rows 64t..64t+63]
    TSS_CU(cudaMemset(tmp, 0, gu_rows * d * b2));
    for (int t = 0; t < c->Ft; ++t) {
      const int rows = F - 64 * t < 64 ? F - 64 * t : 64;
      const size_t src_off = static_cast<size_t>(64) * t * d;
      TSS_CU(cudaMemcpy(tmp + static_cast<size_t>(t) * 128 * d, static_cast<const __nv_bfloat16*>(w->w_gate[l]) + src_off,
                        static_cast<size_t>(rows) * d * b2, cudaMemcpyDeviceToDevice));
      TSS_CU(cudaMemcpy(tmp + (static_cast<size_t>(t) * 128 + 64) * d, static_cast<const __nv_bfloat16*>(w->w_up[l]) + src_off,
                        static_cast<size_t>(rows) * d * b2, cudaMemcpyDeviceToDevice));
    }
    TSS_CU(launch_tile_weights(tmp, c->wgu + static_cast<size_t>(l) * gu_rows * d, static_cast<int>(gu_rows), d, 0));
    TSS_CU(cudaMemset(tmp, 0, static_cast<size_t>(d) * c->F_pad * b2));
    TSS_CU(cudaMemcpy2D(tmp, static_cast<size_t>(c->F_pad) * b2, w->w_down[l], static_cast<size_t>(F) * b2,
                        static_cast<size_t>(F) * b2, d, cudaMemcpyDeviceToDevice));
    TSS_CU(launch_tile_weights(tmp, c->wdown + static_cast<size_t>(l) * d * c->F_pad, d, c->F_pad, 0));
    TSS_CU(launch_bf16_to_f32(static_cast<const __nv_bfloat16*>(w->attn_norm[l]), c->g_attn + static_cast<size_t>(l) * d, d, 0));
    TSS_CU(launch_bf16_to_f32(static_cast<const __nv_bfloat16*>(w->mlp_norm[l]), c->g_mlp + static_cast<size_t>(l) * d, d, 0));
    TSS_CU(cudaDeviceSynchronize());  // the staging buffer is reused by the next layer
  }
  return TSS_OK;
}

tss_status build_workspaces(tss_ctx* c) {
  const int d = c->d;
  const size_t R = kMaxRows;
  TSS_TRY(c->alloc(&c->h, R * d));
  TSS_TRY(c->alloc(&c->xn, 2 * R * d));  // persistent path: hi and lo parts
  TSS_TRY(c->alloc(&c->qbuf, R * d));
  TSS_TRY(c->alloc(&c->obuf, 2 * R * d));
  TSS_TRY(c->alloc(&c->act, 2 * R * c->F_pad));
  TSS_TRY(c->alloc(&c->logits_ws, static_cast<size_t>(c->a.max_rows) * c->V));
  TSS_CU(cudaMemset(c->xn, 0, 2 * R * d * 2));
  TSS_CU(cudaMemset(c->obuf, 0, 2 * R * d * 2));
  TSS_CU(cudaMemset(c->act, 0, 2 * R * c->F_pad * 2));
  const int max_tiles = std::max(std::max(3 * d / 128, c->Ft), c->V_pad / 128);
  const size_t max_grid = static_cast<size_t>(c->num_sms) * 2;
  c->partials_floats = (max_grid + max_tiles) * 128 * static_cast<size_t>(pad_to(c->a.max_rows, 16));
  TSS_TRY(c->alloc(&c->partials, c->partials_floats));
  TSS_TRY(c->alloc(&c->counters, max_tiles + 64));
  TSS_CU(cudaMemset(c->counters, 0, (max_tiles + 64) * sizeof(int)));
  TSS_TRY(c->alloc(&c->amax_val, static_cast<size_t>(c->V_pad / 128) * kMaxRows));
  TSS_TRY(c->alloc(&c->amax_idx, static_cast<size_t>(c->V_pad / 128) * kMaxRows));
  // partials of the split attention: 64 rows per (request, head, split), 128 for wide blocks
  const size_t ph = static_cast<size_t>(c->a.max_batch) * c->H * c->max_splits *
                    (c->a.max_nodes > kNarrowNodes ? kMaxNodes : kNarrowNodes);
  TSS_TRY(c->alloc(&c->attn_po, ph * c->D));
  TSS_TRY(c->alloc(&c->attn_pml, ph * 2));
  if (c->D == 128 && c->attn_tc) {
    TSS_TRY(c->alloc(&c->d_kvmaps, c->L));
    c->h_kvmaps.assign(c->L, CUtensorMap{});
    c->kvmap_ptr.assign(c->L, nullptr);
    const size_t tr = attn_tc_partial_rows(c->a.max_batch, c->H, c->num_sms);
    TSS_TRY(c->alloc(&c->tc_po, tr * 128));
    TSS_TRY(c->alloc(&c->tc_pml, tr * 2));
  }
  TSS_TRY(c->alloc(&c->d_step, 1));
  TSS_TRY(c->alloc(&c->d_plan, 1));
  TSS_CU(cudaMemset(c->d_plan, 0, sizeof(PlanDev)));
  c->phi.assign(c->a.max_domains, 0ull);
  c->phi_valid.assign(c->a.max_domains, 0);
  TSS_TRY(c->alloc(&c->d_status, 1));
  TSS_CU(cudaMemset(c->d_status, 0, sizeof(int)));
  TSS_CU(cudaMallocHost(&c->h_status, sizeof(int)));
  for (int i = 0; i < kRing; ++i) {
    TSS_CU(cudaMallocHost(&c->h_ring[i], sizeof(StepDesc)));
    TSS_CU(cudaEventCreateWithFlags(&c->ring_ev[i], cudaEventDisableTiming));
  }
  TSS_TRY(c->alloc(&c->io_tokens, kMaxRows));
  TSS_TRY(c->alloc(&c->io_probs, static_cast<size_t>(c->a.max_rows) * c->V));
  TSS_TRY(c->alloc(&c->io_unif, static_cast<size_t>(c->a.max_batch) * 4 * kMaxNodes));
  TSS_TRY(c->alloc(&c->io_res, static_cast<size_t>(kMaxBatch) * (3 + kMaxPathStride)));
  // RoPE tables in float64, stored as float32: angle(pos, i) = pos * theta^(-2i/D)
  const int half = c->D / 2;
  std::vector<float> hc(static_cast<size_t>(c->a.max_positions) * half), hs(hc.size());
  for (int pos = 0; pos < c->a.max_positions; ++pos)
    for (int i = 0; i < half; ++i) {
      const double inv = std::pow(static_cast<double>(c->a.rope_theta), -2.0 * i / c->D);
      const double ang = static_cast<double>(pos) * inv;
      hc[static_cast<size_t>(pos) * half + i] = static_cast<float>(std::cos(ang));
      hs[static_cast<size_t>(pos) * half + i] = static_cast<float>(std::sin(ang));
    }
  TSS_TRY(c->alloc(&c->rope_cos, hc.size()));
  TSS_TRY(c->alloc(&c->rope_sin, hs.size()));
  TSS_CU(cudaMemcpy(c->rope_cos, hc.data(), hc.size() * 4, cudaMemcpyHostToDevice));
  TSS_CU(cudaMemcpy(c->rope_sin, hs.data(), hs.size() * 4, cudaMemcpyHostToDevice));
  TSS_CU(cudaStreamCreateWithFlags(&c->cap_stream, cudaStreamNonBlocking));
  size_t max_smem = gemm_smem_bytes(16, 12);
  for (int n = 16; n <= 256; n += 16) max_smem = std::max(max_smem, gemm_smem_bytes(n, 2));
  max_smem = std::max<size_t>(max_smem, 220 * 1024 + 16 * 1024);
  if (max_smem > 232448) max_smem = 232448;
  TSS_CU(gemm_prepare(max_smem));
  TSS_CU(attn_prepare());
  TSS_CU(attn_tc_prepare());
  TSS_CU(pf_prepare());
  TSS_CU(mk_prepare());
  {
    const int nt = d / 128;
    c->mk_max_tiles = max_tiles;
    TSS_TRY(c->alloc(&c->ssp, static_cast<size_t>(nt) * kMaxRows));
    TSS_CU(cudaMemset(c->ssp, 0, static_cast<size_t>(nt) * kMaxRows * sizeof(float)));
    const size_t nflags = static_cast<size_t>(nt) + 3 * nt + c->Ft + static_cast<size_t>(c->a.max_batch) * c->H;
    TSS_TRY(c->alloc(&c->flags, nflags));
    TSS_CU(cudaMemset(c->flags, 0, nflags * sizeof(unsigned long long)));
    // stream-K counters, the abort word and the attention's split counters: zeroed by every
    // step's prologue, so that a step after one that gave up on a timeout starts clean
    c->mk_n_zero = 7 * max_tiles + 1 + c->a.max_batch * c->H;
    TSS_TRY(c->alloc(&c->mk_zero, static_cast<size_t>(c->mk_n_zero)));
    TSS_CU(cudaMemset(c->mk_zero, 0, static_cast<size_t>(c->mk_n_zero) * sizeof(int)));
    c->attn_cnt = c->mk_zero + 7 * max_tiles + 1;
    // partial tiles are strided by the MMA width of the split B operand (up to 256 rows)
    int xs_rows_max = 16;
    for (int m = 1; m <= c->a.max_rows; ++m) xs_rows_max = std::max(xs_rows_max, xs_layout(m).rows);
    c->mk_part_floats = (static_cast<size_t>(c->num_sms) + max_tiles) * 128 * static_cast<size_t>(xs_rows_max);
    TSS_TRY(c->alloc(&c->mk_part0, c->mk_part_floats));
    TSS_TRY(c->alloc(&c->mk_part1, c->mk_part_floats));
  }
  TSS_CU(misc_prepare());
  return TSS_OK;
}

void destroy_ctx(tss_ctx* c) {
  if (!c) return;
  for (auto& kv : c->graphs) cudaGraphExecDestroy(kv.second);
  for (void* p : c->allocs) cudaFree(p);
  for (int i = 0; i < kRing; ++i) {
    if (c->h_ring[i]) cudaFreeHost(c->h_ring[i]);
    if (c->ring_ev[i]) cudaEventDestroy(c->ring_ev[i]);
  }
  if (c->h_status) cudaFreeHost(c->h_status);
  if (c->cap_stream) cudaStreamDestroy(c->cap_stream);
  delete c;
}

// Host-side per-step checks and the descriptor contents.  Nothing is enqueued here.
// rng_ids (optional): the Philox request index of each request (default: its index in the batch).
tss_status prepare_step(const tss_ctx* c, const tss_verify_batch* bt, const tss_kv_cache* kv,
                        const tss_verify_result* res, StepDesc* sd, StepPlan* sp, const int* rng_ids = nullptr) {
  if (!bt || !kv || !res) return fail(TSS_ERR_INVALID_ARG, "batch, kv or result is NULL");
  const int B = bt->n_req;
  if (B < 1 || B > c->a.max_batch) return fail(TSS_ERR_INVALID_ARG, "n_req must be in [1, max_batch]");
  if (!bt->n_nodes || !bt->ctx_len || !bt->domain_id || !bt->parent_idx || !bt->tokens)
    return fail(TSS_ERR_INVALID_ARG, "n_nodes, ctx_len, domain_id, parent_idx and tokens are required");
  if (bt->mode != TSS_MODE_GREEDY && bt->mode != TSS_MODE_SAMPLE) return fail(TSS_ERR_INVALID_ARG, "unknown mode");
  if (!kv->layer || kv->n_slots < 1 || kv->cap < 1) return fail(TSS_ERR_INVALID_ARG, "KV cache descriptor invalid");
  if (!res->accept_len || !res->bonus || !res->path || !res->new_ctx_len)
    return fail(TSS_ERR_INVALID_ARG, "result arrays accept_len, bonus, path and new_ctx_len are required");
  std::memset(sd, 0, sizeof(StepDesc));
  int M = 0, max_depth = 0, max_t = 0;
  std::vector<int> slot_used(kv->n_slots, 0);
  unsigned long long all_runs = 0ull;  // layers some request runs
  for (int b = 0; b < B; ++b) {
    const int n = bt->n_nodes[b], ctx = bt->ctx_len[b];
    if (n < 1 || n > c->a.max_nodes) return fail(TSS_ERR_INVALID_ARG, "n_nodes out of [1, max_nodes]");
    if (M + n > c->a.max_rows) return fail(TSS_ERR_INVALID_ARG, "total rows exceed max_rows");
    if (ctx < 0) return fail(TSS_ERR_INVALID_ARG, "ctx_len negative");
    if (static_cast<long long>(ctx) + n > kv->cap) return fail(TSS_ERR_KV_CAPACITY, "ctx_len + n_nodes exceeds KV capacity");
    const int slot = bt->kv_slot ? bt->kv_slot[b] : b;
    if (slot < 0 || slot >= kv->n_slots) return fail(TSS_ERR_INVALID_ARG, "kv_slot out of range");
    if (slot_used[slot]++) return fail(TSS_ERR_INVALID_ARG, "two requests share a kv_slot");
    const int dom = bt->domain_id[b];
    const bool configured = dom >= 0 && dom < c->a.max_domains && c->phi_valid[dom];
    const unsigned long long mask = configured ? c->phi[dom] : 0ull;  // S(x) or dense fallback
    for (int l = 0; l < c->L; ++l)
      if (!((mask >> l) & 1ull)) all_runs |= 1ull << l;
    sd->req_ctx[b] = ctx;
    sd->req_nodes[b] = n;
    sd->req_rowoff[b] = M;
    sd->req_slot[b] = slot;
    sd->req_domain[b] = dom;
    sd->req_rng[b] = rng_ids ? rng_ids[b] : b;
    sd->req_phi[b] = mask;
    unsigned long long anc[kMaxNodes], anc_hi[kMaxNodes];  // ancestor-or-self bits of rows 0..63, 64..127
    int depth[kMaxNodes];
    for (int i = 0; i < n; ++i) {
      const int par = bt->parent_idx[M + i];
      if (i == 0 ? par != -1 : (par < 0 || par >= i))
        return fail(TSS_ERR_INVALID_ARG, "parent_idx must be -1 for row 0 and in [0, i) otherwise");
      if (bt->mode == TSS_MODE_SAMPLE && i > 0 && par != i - 1)
        return fail(TSS_ERR_INVALID_ARG, "speculative sampling verifies chain drafts only");
      depth[i] = i == 0 ? 0 : depth[par] + 1;
      anc[i] = (i == 0 ? 0ull : anc[par]) | (i < 64 ? 1ull << i : 0ull);
      anc_hi[i] = (i == 0 ? 0ull : anc_hi[par]) | (i >= 64 ? 1ull << (i - 64) : 0ull);
      const int pos = ctx + depth[i];
      if (bt->positions && bt->positions[M + i] != pos)
        return fail(TSS_ERR_INVALID_ARG, "positions must equal ctx_len + depth");
      if (pos >= c->a.max_positions) return fail(TSS_ERR_INVALID_ARG, "position beyond max_positions");
      sd->row_req[M + i] = b;
      sd->row_pos[M + i] = pos;
      sd->row_parent[M + i] = par;
      sd->row_anc[M + i] = anc[i];
      sd->row_anc_hi[M + i] = anc_hi[i];
      if (depth[i] > max_depth) max_depth = depth[i];
    }
    max_t = std::max(max_t, ctx + n);
    M += n;
  }
  if (res->path_stride < max_depth + 1 || res->path_stride > kMaxPathStride)
    return fail(TSS_ERR_INVALID_ARG, "path_stride must be in [max depth + 1, 1024]");
  for (int l = 0; l < c->L; ++l)
    if (((all_runs >> l) & 1ull)) {
      if (!kv->layer[l]) return fail(TSS_ERR_INVALID_ARG, "KV buffer of an active layer is NULL");
      if (!aligned16(kv->layer[l])) return fail(TSS_ERR_INVALID_ARG, "KV buffers must be 16-byte aligned");
    }
  if (bt->mode == TSS_MODE_SAMPLE) {
    if (!(bt->temperature > 0.f) || !std::isfinite(bt->temperature))
      return fail(TSS_ERR_INVALID_ARG, "temperature must be positive and finite");
    if (!bt->draft_probs) return fail(TSS_ERR_INVALID_ARG, "draft_probs required for speculative sampling");
    if (bt->uniforms) {
      int need = 0;
      for (int b = 0; b < B; ++b) need = std::max(need, 2 * (bt->n_nodes[b] - 1) + 1);
      if (bt->uniform_stride < need) return fail(TSS_ERR_INVALID_ARG, "uniform_stride < 2k + 1");
      if (bt->io_host && bt->uniform_stride > 4 * kMaxNodes)
        return fail(TSS_ERR_INVALID_ARG, "uniform_stride too large for host I/O");
    }
  }
  int n_act = 0;
  for (int l = 0; l < c->L; ++l) n_act += (all_runs >> l) & 1ull;
  sd->B = B;
  sd->M = M;
  sd->n_act_host = n_act;
  sd->mode = bt->mode;
  sd->inv_temperature = bt->mode == TSS_MODE_SAMPLE ? 1.f / bt->temperature : 1.f;
  sd->uniform_stride = bt->uniform_stride;
  sd->path_stride = res->path_stride;
  sd->kv_cap = kv->cap;
  sd->seed_lo = static_cast<uint32_t>(bt->philox_seed);
  sd->seed_hi = static_cast<uint32_t>(bt->philox_seed >> 32);
  sd->off_lo = static_cast<uint32_t>(bt->philox_offset);
  sd->off_hi = static_cast<uint32_t>(bt->philox_offset >> 32);
  for (int l = 0; l < c->L; ++l) sd->kv_layer[l] = static_cast<__nv_bfloat16*>(kv->layer[l]);
  const int tiles = (max_t + 63) / 64;
  const int splits = c->attn_splits_force > 0 ? std::min(c->attn_splits_force, c->max_splits) : ext_attn_splits(c, sd, B);
  sp->B = B;
  sp->M = M;
  sp->n_act = n_act;
  sp->mode = bt->mode;
  sp->splits = splits;
  sp->n_pad = pad_to(M, 16);
  sp->max_nodes = 1;
  for (int b = 0; b < B; ++b) sp->max_nodes = std::max(sp->max_nodes, bt->n_nodes[b]);
  sp->tiles = tiles;
  sp->ctx_sum = 0;
  for (int b = 0; b < B; ++b) sp->ctx_sum += bt->ctx_len[b];
  return TSS_OK;
}

// Workspaces of the compute-bound prefill, made at the first call: passes of up to 4096 rows.
tss_status pf_workspaces(tss_ctx* c) {
  if (c->pf_tmax) return TSS_OK;
  const int T = 4096;
  const size_t d = c->d, F = c->F_pad;
  TSS_TRY(c->alloc(&c->pf_h, T * d));
  TSS_TRY(c->alloc(&c->pf_xh, T * d));
  TSS_TRY(c->alloc(&c->pf_xl, T * d));
  TSS_TRY(c->alloc(&c->pf_qh, T * d));
  TSS_TRY(c->alloc(&c->pf_ql, T * d));
  TSS_TRY(c->alloc(&c->pf_ah, T * d));
  TSS_TRY(c->alloc(&c->pf_al, T * d));
  TSS_TRY(c->alloc(&c->pf_uh, T * F));
  TSS_TRY(c->alloc(&c->pf_ul, T * F));
  TSS_TRY(c->alloc(&c->pf_tok, T));
  TSS_TRY(c->alloc(&c->pf_pos, T));
  TSS_TRY(c->alloc(&c->pf_slot, T));
  TSS_TRY(c->alloc(&c->pf_qt, T / 128));
  // (rows past a pass's rows are read by the last tile of each GEMM and attention: finite)
  TSS_CU(cudaMemset(c->pf_xh, 0, T * d * 2));
  TSS_CU(cudaMemset(c->pf_xl, 0, T * d * 2));
  TSS_CU(cudaMemset(c->pf_qh, 0, T * d * 2));
  TSS_CU(cudaMemset(c->pf_ql, 0, T * d * 2));
  TSS_CU(cudaMemset(c->pf_ah, 0, T * d * 2));
  TSS_CU(cudaMemset(c->pf_al, 0, T * d * 2));
  TSS_CU(cudaMemset(c->pf_uh, 0, T * F * 2));
  TSS_CU(cudaMemset(c->pf_ul, 0, T * F * 2));
  const struct {
    CUtensorMap* m;
    const void* p;
    size_t k;
  } maps[] = {{&c->pf_tm_xh, c->pf_xh, d}, {&c->pf_tm_xl, c->pf_xl, d}, {&c->pf_tm_qh, c->pf_qh, d},
              {&c->pf_tm_ql, c->pf_ql, d}, {&c->pf_tm_ah, c->pf_ah, d}, {&c->pf_tm_al, c->pf_al, d},
              {&c->pf_tm_uh, c->pf_uh, F}, {&c->pf_tm_ul, c->pf_ul, F}};
  for (const auto& m : maps)
    if (!make_tmap(m.m, m.p, m.k, T, 1, 128, 2)) return fail(TSS_ERR_CUDA, "cuTensorMapEncodeTiled failed (prefill)");
  c->pf_tmax = T;
  return TSS_OK;
}

// One pass: T rows (the row tables and tokens already in place) through every layer the skip set
// keeps (Sec. "Domain-Aware Skip Controller": h_{l+1} = h_l for a skipped layer, which writes no KV).
tss_status pf_pass(tss_ctx* c, int T, int n_qtiles, unsigned long long skip, const tss_kv_cache* kv, cudaStream_t s,
                   bool inject) {
  PfParams p{};
  p.T = T;
  p.n_qtiles = n_qtiles;
  p.d_model = c->d;
  p.n_heads = c->H;
  p.head_dim = c->D;
  p.vocab = c->V;
  p.kv_cap = kv->cap;
  p.row_pos = c->pf_pos;
  p.row_slot = c->pf_slot;
  p.qtiles = c->pf_qt;
  p.rms_eps = c->a.rms_eps;
  p.tokens = c->pf_tok;
  p.embed = c->embed;
  p.h = c->pf_h;
  p.xh = c->pf_xh;
  p.xl = c->pf_xl;
  p.x_ld = c->d;
  p.qh = c->pf_qh;
  p.ql = c->pf_ql;
  p.ah = c->pf_ah;
  p.al = c->pf_al;
  p.uh = c->pf_uh;
  p.ul = c->pf_ul;
  p.u_ld = c->F_pad;
  p.rope_cos = c->rope_cos;
  p.rope_sin = c->rope_sin;
  p.status = c->d_status;
  const unsigned long long rows = static_cast<unsigned long long>(kv->n_slots) * 2ull * c->H * kv->cap;
  if (rows + 64 > 0x7fffffffull) return fail(TSS_ERR_INVALID_ARG, "KV cache too large for the prefill's tensor maps");
  TSS_CU(launch_pf_embed(p, s));
  const int d = c->d, kbd = d / 64, G = c->num_sms;
  const size_t dd = static_cast<size_t>(d) * d;
  for (int l = 0; l < c->L; ++l) {
    if ((skip >> l) & 1ull) continue;
    CUtensorMap tkv;
    if (!make_tmap(&tkv, kv->layer[l], 128, rows, 1, 64, 2)) return fail(TSS_ERR_CUDA, "cuTensorMapEncodeTiled failed (prefill KV)");
    p.kv = static_cast<__nv_bfloat16*>(kv->layer[l]);
    TSS_CU(launch_pf_norm(p, c->g_attn + static_cast<size_t>(l) * d, s));
    TSS_CU(launch_pf_gemm(kPfEpiQkv, c->pf_tm_xh, c->pf_tm_xl, p,
                          PfGemm{c->wqkv, static_cast<long long>(3 * dd), l, 3 * d / 128, kbd, inject ? 1 : 0}, G, s));
    inject = false;
    TSS_CU(launch_pf_attn(c->pf_tm_qh, c->pf_tm_ql, tkv, p, s));
    TSS_CU(launch_pf_gemm(kPfEpiResid, c->pf_tm_ah, c->pf_tm_al, p, PfGemm{c->wo, static_cast<long long>(dd), l, d / 128, kbd, 0}, G, s));
    TSS_CU(launch_pf_norm(p, c->g_mlp + static_cast<size_t>(l) * d, s));
    TSS_CU(launch_pf_gemm(kPfEpiSwiglu, c->pf_tm_xh, c->pf_tm_xl, p,
                          PfGemm{c->wgu, static_cast<long long>(c->Ft) * 128 * d, l, c->Ft, kbd, 0}, G, s));
    TSS_CU(launch_pf_gemm(kPfEpiResid, c->pf_tm_uh, c->pf_tm_ul, p,
                          PfGemm{c->wdown, static_cast<long long>(d) * c->F_pad, l, d / 128, c->F_pad / 64, 0}, G, s));
  }
  return TSS_OK;
}

}  // namespace

extern "C" {

const char* tss_status_string(tss_status s) {
  switch (s) {
    case TSS_OK: return "ok";
    case TSS_ERR_INVALID_ARG: return "invalid argument";
    case TSS_ERR_OUT_OF_MEMORY: return "out of device memory";
    case TSS_ERR_KV_CAPACITY: return "KV cache capacity exceeded";
    case TSS_ERR_CUDA: return "CUDA error";
    case TSS_ERR_UNSUPPORTED_ARCH: return "unsupported model shape or GPU";
    case TSS_ERR_TIMEOUT: return "device wait timed out";
    case TSS_ERR_DEVICE_CHECK: return "device-side check failed";
    default: return "unknown status";
  }
}

const char* tss_last_error(void) { return g_err.c_str(); }

int tss_attention_kernel(const tss_ctx* c) { return c ? c->last_attn : -1; }

tss_status tss_create(const tss_weights* weights, const tss_arch* arch, tss_ctx** out) {
  if (!out) return fail(TSS_ERR_INVALID_ARG, "out is NULL");
  *out = nullptr;
  TSS_TRY(validate_arch(arch));
  int dev = 0;
  TSS_CU(cudaGetDevice(&dev));
  cudaDeviceProp prop;
  TSS_CU(cudaGetDeviceProperties(&prop, dev));
  if (prop.major != 10 || prop.minor != 3)
    return fail(TSS_ERR_UNSUPPORTED_ARCH, "this library is built for sm_103 (GB300); device is sm_" +
                                               std::to_string(prop.major) + std::to_string(prop.minor));
  if (!encode_fn()) return fail(TSS_ERR_CUDA, "cuTensorMapEncodeTiled unavailable");
  tss_ctx* c = new tss_ctx();
  c->a = *arch;
  c->dev = dev;
  c->num_sms = prop.multiProcessorCount;
  c->L = arch->n_layers;
  c->d = arch->d_model;
  c->H = arch->n_heads;
  c->D = arch->head_dim;
  c->F = arch->d_mlp;
  c->V = arch->vocab;
  c->Ft = (c->F + 63) / 64;
  c->F_pad = c->Ft * 64;
  c->V_pad = pad_to(c->V, 128);
  if (const char* e = std::getenv("TSS_NO_GRAPH")) c->use_graphs = std::atoi(e) == 0;
  if (const char* e = std::getenv("TSS_GEMM_CTAS_PER_SM")) c->gemm_ctas_per_sm = std::max(1, std::min(2, std::atoi(e)));
  if (const char* e = std::getenv("TSS_PATH")) c->use_mk = std::string(e) != "multi";
  if (const char* e = std::getenv("TSS_ATTN")) {
    const std::string v(e);
    c->attn_mode = v == "internal" ? 1 : v == "external" ? 2 : 0;
  }
  if (const char* e = std::getenv("TSS_MK_KPS")) c->mk_kps = std::min(8, std::max(1, std::atoi(e)));
  if (const char* e = std::getenv("TSS_EVICT_FIRST")) c->w_evict_first = std::atoi(e) != 0;
  if (const char* e = std::getenv("TSS_ATTN_PLO")) c->attn_plo = std::atoi(e) != 0;
  if (const char* e = std::getenv("TSS_ATTN_SPLITS")) c->attn_splits_force = std::max(0, std::atoi(e));
  if (const char* e = std::getenv("TSS_ATTN_TC")) c->attn_tc = std::atoi(e) != 0;
  if (const char* e = std::getenv("TSS_MK_ATTN_SPLITS")) c->mk_splits_force = std::max(0, std::atoi(e));
  if (const char* e = std::getenv("TSS_PREFILL")) c->pf_enabled = std::string(e) != "steps";
  if (const char* e = std::getenv("TSS_MK_STAGES")) c->mk_max_stages = std::min(12, std::max(2, std::atoi(e)));
  if (const char* e = std::getenv("TSS_MK_DP")) c->mk_dp_tail = std::atoi(e) != 0;
  if (const char* e = std::getenv("TSS_ALLOC_LIMIT_BYTES")) c->alloc_limit = std::strtoull(e, nullptr, 10);
  if (const char* e = std::getenv("TSS_WAIT_LIMIT_MS")) {
    const long long ms = std::atoll(e);
    if (ms >= 1 && ms <= 600000) c->wait_ns = static_cast<unsigned long long>(ms) * 1000000ull;
  }
  const char* trace_env = std::getenv("TSS_TRACE");
  tss_status s = build_workspaces(c);
  if (s == TSS_OK) s = build_weights(c, weights);
  if (s == TSS_OK && trace_env && std::atoi(trace_env) != 0) {
    s = c->alloc(&c->trace, static_cast<size_t>(c->num_sms) * mk_trace_slots());
    if (s == TSS_OK && cudaMemset(c->trace, 0, static_cast<size_t>(c->num_sms) * mk_trace_slots() * 8) != cudaSuccess)
      s = fail(TSS_ERR_CUDA, "cudaMemset of the trace buffer failed");
  }
  if (s != TSS_OK) {
    const std::string msg = g_err;
    destroy_ctx(c);
    cudaGetLastError();
    g_err = msg;
    return s;
  }
  *out = c;
  return TSS_OK;
}

void tss_destroy(tss_ctx* ctx) {
  if (!ctx) return;
  cudaDeviceSynchronize();
  destroy_ctx(ctx);
}

tss_status tss_set_skip_config(tss_ctx* c, int domain_id, uint64_t mask) {
  if (!c) return fail(TSS_ERR_INVALID_ARG, "ctx is NULL");
  if (domain_id < 0 || domain_id >= c->a.max_domains) return fail(TSS_ERR_INVALID_ARG, "domain_id out of range");
  if (c->L < 64 && (mask >> c->L) != 0ull) return fail(TSS_ERR_INVALID_ARG, "skip mask names a layer >= n_layers");
  // Host-only: a step takes each request's S(x) from this map when it is enqueued (into its
  // descriptor), so steps already enqueued keep the map they were planned with and nothing waits.
  c->phi[domain_id] = mask;
  c->phi_valid[domain_id] = 1;
  return TSS_OK;
}

tss_status tss_clear_skip_config(tss_ctx* c, int domain_id) {
  if (!c) return fail(TSS_ERR_INVALID_ARG, "ctx is NULL");
  if (domain_id < 0 || domain_id >= c->a.max_domains) return fail(TSS_ERR_INVALID_ARG, "domain_id out of range");
  c->phi[domain_id] = 0ull;  // host-only, as in tss_set_skip_config
  c->phi_valid[domain_id] = 0;
  return TSS_OK;
}

tss_status tss_sparsity_ratio(const tss_ctx* c, int domain_id, double* out) {
  if (!c || !out) return fail(TSS_ERR_INVALID_ARG, "ctx or out is NULL");
  if (domain_id < 0 || domain_id >= c->a.max_domains) return fail(TSS_ERR_INVALID_ARG, "domain_id out of range");
  const unsigned long long m = c->phi_valid[domain_id] ? c->phi[domain_id] : 0ull;
  *out = static_cast<double>(__builtin_popcountll(m)) / c->L;
  return TSS_OK;
}

tss_status tss_estimate_step_bytes(const tss_arch* a, int n_req, const uint64_t* masks, const int32_t* ctx_len,
                                   const int32_t* n_nodes, tss_step_bytes* out) {
  if (!a || !masks || !ctx_len || !n_nodes || !out) return fail(TSS_ERR_INVALID_ARG, "NULL argument");
  if (n_req < 1) return fail(TSS_ERR_INVALID_ARG, "n_req must be positive");
  if (a->n_layers < 1 || a->n_layers > 64 || a->d_model < 1 || a->d_mlp < 1 || a->vocab < 1)
    return fail(TSS_ERR_INVALID_ARG, "arch: n_layers in [1, 64], positive d_model, d_mlp and vocab");
  const int L = a->n_layers;
  const uint64_t d = static_cast<uint64_t>(a->d_model), f = static_cast<uint64_t>(a->d_mlp);
  const uint64_t kv_token = 4 * d;  // K and V rows of one token in one layer, bf16
  uint64_t runs = 0, kv_read = 0, kv_write = 0;
  for (int b = 0; b < n_req; ++b) {
    if (L < 64 && (masks[b] >> L) != 0) return fail(TSS_ERR_INVALID_ARG, "a skip mask names a layer >= n_layers");
    if (ctx_len[b] < 0 || n_nodes[b] < 0) return fail(TSS_ERR_INVALID_ARG, "ctx_len and n_nodes must be >= 0");
    const uint64_t all = L == 64 ? ~0ull : (1ull << L) - 1;
    const uint64_t act = all & ~masks[b];
    runs |= act;
    const uint64_t n_act = static_cast<uint64_t>(__builtin_popcountll(act));
    kv_read += static_cast<uint64_t>(ctx_len[b]) * n_act * kv_token;
    kv_write += static_cast<uint64_t>(n_nodes[b]) * n_act * kv_token;
  }
  out->active_union = __builtin_popcountll(runs);
  out->weights = static_cast<uint64_t>(out->active_union) * 2 * (4 * d * d + 3 * d * f) +
                 static_cast<uint64_t>(a->vocab) * d * 2;
  out->kv_read = kv_read;
  out->kv_write = kv_write;
  out->total = out->weights + kv_read + kv_write;
  return TSS_OK;
}

tss_status tss_persistent_plan(const tss_arch* a, int n_req, int n_rows, int max_keys, int num_sms,
                               tss_persistent_plan_info* out) {
  if (!a || !out) return fail(TSS_ERR_INVALID_ARG, "NULL argument");
  if ((a->head_dim != 64 && a->head_dim != 128) || a->n_heads < 1)
    return fail(TSS_ERR_INVALID_ARG, "arch: head_dim 64 or 128 and n_heads >= 1");
  if (n_req < 1 || n_req > kMaxBatch || n_rows < n_req || n_rows > kMaxRows || max_keys < 1 || num_sms < 1)
    return fail(TSS_ERR_INVALID_ARG, "n_req in [1, 64], n_rows in [n_req, 256], max_keys and num_sms positive");
  const MkPlanIn in{a->head_dim, a->n_heads, num_sms, 3, 12, kMaxSplits, 0};
  MkConfig cfg;
  const bool fits = mk_config_for(in, n_req, n_rows, (max_keys + 63) / 64, &cfg);
  out->fits = fits ? 1 : 0;
  out->kps = fits ? cfg.kps : 0;
  out->stages = fits ? cfg.stages : 0;
  out->attn_splits = fits ? cfg.attn_splits : 0;
  out->smem_bytes = fits ? static_cast<uint64_t>(cfg.smem) : 0;
  return TSS_OK;
}

tss_status tss_active_layer_count(const tss_ctx* c, const tss_verify_batch* bt, int* out) {
  if (!c || !bt || !out || !bt->domain_id) return fail(TSS_ERR_INVALID_ARG, "NULL argument");
  if (bt->n_req < 1 || bt->n_req > c->a.max_batch) return fail(TSS_ERR_INVALID_ARG, "n_req out of range");
  unsigned long long runs = 0ull;
  for (int b = 0; b < bt->n_req; ++b) {
    const int dom = bt->domain_id[b];
    const unsigned long long m = (dom >= 0 && dom < c->a.max_domains && c->phi_valid[dom]) ? c->phi[dom] : 0ull;
    for (int l = 0; l < c->L; ++l)
      if (!((m >> l) & 1ull)) runs |= 1ull << l;
  }
  *out = __builtin_popcountll(runs);
  return TSS_OK;
}

}  // extern "C"

namespace {

tss_status verify_impl(tss_ctx* c, const tss_verify_batch* bt, const tss_kv_cache* kv, const tss_verify_result* res,
                       cudaStream_t s, Prof* prof, const int* rng_ids = nullptr) {
  if (!c) return fail(TSS_ERR_INVALID_ARG, "ctx is NULL");
  const int ri = c->ring_i;
  if (c->ring_used[ri]) TSS_CU(cudaEventSynchronize(c->ring_ev[ri]));
  StepDesc* sd = c->h_ring[ri];
  StepPlan sp;
  TSS_TRY(prepare_step(c, bt, kv, res, sd, &sp, rng_ids));
  const int M = sp.M, B = sp.B;
  const bool host_io = bt->io_host != 0;
  if (host_io) {
    sd->tokens = c->io_tokens;
    sd->draft_probs = bt->mode == TSS_MODE_SAMPLE ? c->io_probs : nullptr;
    sd->uniforms = (bt->mode == TSS_MODE_SAMPLE && bt->uniforms) ? c->io_unif : nullptr;
    sd->accept_len = c->io_res;
    sd->bonus = c->io_res + kMaxBatch;
    sd->new_ctx = c->io_res + 2 * kMaxBatch;
    sd->path = c->io_res + 3 * kMaxBatch;
  } else {
    sd->tokens = bt->tokens;
    sd->draft_probs = bt->draft_probs;
    sd->uniforms = bt->uniforms;
    sd->accept_len = res->accept_len;
    sd->bonus = res->bonus;
    sd->new_ctx = res->new_ctx_len;
    sd->path = res->path;
  }
  // logits: the caller's buffer, else (sampling needs them) the workspace, else none
  float* logits_dev = (res->logits && !host_io) ? res->logits : nullptr;
  if (!logits_dev && (bt->mode == TSS_MODE_SAMPLE || (host_io && res->logits))) logits_dev = c->logits_ws;
  sd->logits = logits_dev;

  TSS_CU(cudaMemcpyAsync(c->d_step, sd, sizeof(StepDesc), cudaMemcpyHostToDevice, s));
  TSS_TRY(sync_kv_maps(c, kv, s));
  TSS_CU(cudaEventRecord(c->ring_ev[ri], s));
  c->ring_used[ri] = true;
  c->ring_i = (ri + 1) % kRing;
  if (host_io) {
    TSS_CU(cudaMemcpyAsync(c->io_tokens, bt->tokens, sizeof(int) * M, cudaMemcpyHostToDevice, s));
    if (bt->mode == TSS_MODE_SAMPLE) {
      TSS_CU(cudaMemcpyAsync(c->io_probs, bt->draft_probs, sizeof(float) * M * c->V, cudaMemcpyHostToDevice, s));
      if (bt->uniforms)
        TSS_CU(cudaMemcpyAsync(c->io_unif, bt->uniforms, sizeof(float) * B * bt->uniform_stride, cudaMemcpyHostToDevice, s));
    }
  }
  const bool mk = mk_supported(c, sp);
  if (c->use_mk && !mk)
    return fail(TSS_ERR_UNSUPPORTED_ARCH,
                "the step does not fit the persistent kernel's shared-memory plan (and the kernel-per-operation path, "
                "TSS_PATH=multi, does not meet the logit tolerance at 7B/13B widths)");
  if (mk) {
    // Persistent path: three launches per step (the verify kernel is a cooperative launch), so no
    // graph is needed; with a Prof the events bracket each launch directly.
    if (prof) prof->s = s;
    TSS_TRY(enqueue_step_mk(c, sp, s, prof));
  } else if (prof) {
    c->last_attn = attn_variant(c, sp);
    // Launches bracketed by events, captured into a graph so that the device runs them back to
    // back: the events then time device work only, not host launch latency.
    prof->s = c->cap_stream;
    prof->capturing = true;
    cudaGraph_t graph = nullptr;
    TSS_CU(cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeThreadLocal));
    tss_status st = enqueue_step(c, sp, c->cap_stream, prof);
    cudaError_t ce = cudaStreamEndCapture(c->cap_stream, &graph);
    if (st != TSS_OK) {
      if (graph) cudaGraphDestroy(graph);
      return st;
    }
    if (ce != cudaSuccess) return fail(TSS_ERR_CUDA, std::string("profile capture: ") + cudaGetErrorString(ce));
    cudaGraphExec_t exec = nullptr;
    ce = cudaGraphInstantiate(&exec, graph, 0);
    cudaGraphDestroy(graph);
    if (ce != cudaSuccess) return fail(TSS_ERR_CUDA, std::string("profile instantiate: ") + cudaGetErrorString(ce));
    ce = cudaGraphLaunch(exec, s);
    if (ce == cudaSuccess) ce = cudaStreamSynchronize(s);
    cudaGraphExecDestroy(exec);
    if (ce != cudaSuccess) return fail(TSS_ERR_CUDA, std::string("profile launch: ") + cudaGetErrorString(ce));
  } else if (c->use_graphs) {
    c->last_attn = attn_variant(c, sp);
    const GraphKey key{sp.B, sp.M, sp.n_act, sp.mode, sp.splits, attn_variant(c, sp)};
    auto it = c->graphs.find(key);
    if (it == c->graphs.end()) {
      cudaGraph_t graph = nullptr;
      TSS_CU(cudaStreamBeginCapture(c->cap_stream, cudaStreamCaptureModeThreadLocal));
      tss_status st = enqueue_step(c, sp, c->cap_stream);
      cudaError_t ce = cudaStreamEndCapture(c->cap_stream, &graph);
      if (st != TSS_OK) {
        if (graph) cudaGraphDestroy(graph);
        return st;
      }
      if (ce != cudaSuccess) return fail(TSS_ERR_CUDA, std::string("graph capture: ") + cudaGetErrorString(ce));
      cudaGraphExec_t exec = nullptr;
      ce = cudaGraphInstantiate(&exec, graph, 0);
      cudaGraphDestroy(graph);
      if (ce != cudaSuccess) return fail(TSS_ERR_CUDA, std::string("graph instantiate: ") + cudaGetErrorString(ce));
      it = c->graphs.emplace(key, exec).first;
    }
    TSS_CU(cudaGraphLaunch(it->second, s));
  } else {
    c->last_attn = attn_variant(c, sp);
    TSS_TRY(enqueue_step(c, sp, s));
  }
  if (host_io) {
    TSS_CU(cudaMemcpyAsync(res->accept_len, c->io_res, sizeof(int) * B, cudaMemcpyDeviceToHost, s));
    TSS_CU(cudaMemcpyAsync(res->bonus, c->io_res + kMaxBatch, sizeof(int) * B, cudaMemcpyDeviceToHost, s));
    TSS_CU(cudaMemcpyAsync(res->new_ctx_len, c->io_res + 2 * kMaxBatch, sizeof(int) * B, cudaMemcpyDeviceToHost, s));
    TSS_CU(cudaMemcpyAsync(res->path, c->io_res + 3 * kMaxBatch, sizeof(int) * B * res->path_stride,
                           cudaMemcpyDeviceToHost, s));
    if (res->logits)
      TSS_CU(cudaMemcpyAsync(res->logits, c->logits_ws, sizeof(float) * M * c->V, cudaMemcpyDeviceToHost, s));
  }
  return TSS_OK;
}

}  // namespace

extern "C" {

tss_status tss_verify(tss_ctx* c, const tss_verify_batch* bt, const tss_kv_cache* kv, const tss_verify_result* res,
                      void* stream) {
  return verify_impl(c, bt, kv, res, static_cast<cudaStream_t>(stream), nullptr);
}

tss_status tss_verify_grouped(tss_ctx* c, const tss_verify_batch* bt, const tss_kv_cache* kv,
                              const tss_verify_result* res, void* stream, int* n_groups, void* const* group_events) {
  if (!c || !bt || !kv || !res) return fail(TSS_ERR_INVALID_ARG, "ctx, batch, kv or result is NULL");
  if (bt->io_host) return fail(TSS_ERR_INVALID_ARG, "grouped verification takes device arrays (io_host = 0)");
  if (bt->mode == TSS_MODE_SAMPLE && bt->uniforms && bt->uniform_stride > 4 * kMaxNodes)
    return fail(TSS_ERR_INVALID_ARG, "uniform_stride too large for grouped verification");
  // every host-side check of the whole batch first: nothing is enqueued for an invalid batch
  std::vector<StepDesc> scratch(1);
  StepPlan all;
  TSS_TRY(prepare_step(c, bt, kv, res, scratch.data(), &all));
  const int B = bt->n_req;
  const cudaStream_t s = static_cast<cudaStream_t>(stream);
  // groups: requests with the same S(x), fewest active layers first (their requests complete first),
  // ties in order of first appearance
  std::vector<unsigned long long> masks(B);
  std::vector<int> off(B + 1, 0);
  for (int b = 0; b < B; ++b) {
    masks[b] = scratch[0].req_phi[b];
    off[b + 1] = off[b] + bt->n_nodes[b];
  }
  std::vector<unsigned long long> keys;
  for (int b = 0; b < B; ++b)
    if (std::find(keys.begin(), keys.end(), masks[b]) == keys.end()) keys.push_back(masks[b]);
  const uint64_t all_layers = c->L == 64 ? ~0ull : (1ull << c->L) - 1;
  std::stable_sort(keys.begin(), keys.end(), [&](unsigned long long x, unsigned long long y) {
    return __builtin_popcountll(all_layers & ~x) < __builtin_popcountll(all_layers & ~y);
  });
  const size_t V = static_cast<size_t>(c->V);
  for (size_t g = 0; g < keys.size(); ++g) {
    std::vector<int32_t> nn, cl, dom, slot, par, pos;
    std::vector<int> orig;
    int rows = 0;
    for (int b = 0; b < B; ++b) {
      if (masks[b] != keys[g]) continue;
      const int n = bt->n_nodes[b];
      orig.push_back(b);
      nn.push_back(n);
      cl.push_back(bt->ctx_len[b]);
      dom.push_back(bt->domain_id[b]);
      slot.push_back(bt->kv_slot ? bt->kv_slot[b] : b);
      for (int i = 0; i < n; ++i) {
        par.push_back(bt->parent_idx[off[b] + i]);
        if (bt->positions) pos.push_back(bt->positions[off[b] + i]);
      }
      // inputs of the group, contiguous in the context's staging buffers
      TSS_CU(cudaMemcpyAsync(c->io_tokens + rows, bt->tokens + off[b], sizeof(int32_t) * n, cudaMemcpyDeviceToDevice, s));
      if (bt->mode == TSS_MODE_SAMPLE) {
        TSS_CU(cudaMemcpyAsync(c->io_probs + rows * V, bt->draft_probs + off[b] * V, sizeof(float) * n * V,
                               cudaMemcpyDeviceToDevice, s));
        if (bt->uniforms)
          TSS_CU(cudaMemcpyAsync(c->io_unif + (orig.size() - 1) * bt->uniform_stride,
                                 bt->uniforms + static_cast<size_t>(b) * bt->uniform_stride,
                                 sizeof(float) * bt->uniform_stride, cudaMemcpyDeviceToDevice, s));
      }
      rows += n;
    }
    tss_verify_batch sub = *bt;
    sub.n_req = static_cast<int>(nn.size());
    sub.n_nodes = nn.data();
    sub.ctx_len = cl.data();
    sub.domain_id = dom.data();
    sub.kv_slot = slot.data();
    sub.parent_idx = par.data();
    sub.positions = bt->positions ? pos.data() : nullptr;
    sub.tokens = c->io_tokens;
    sub.draft_probs = bt->mode == TSS_MODE_SAMPLE ? c->io_probs : nullptr;
    sub.uniforms = bt->mode == TSS_MODE_SAMPLE && bt->uniforms ? c->io_unif : nullptr;
    tss_verify_result sr{};
    sr.accept_len = c->io_res;
    sr.bonus = c->io_res + kMaxBatch;
    sr.new_ctx_len = c->io_res + 2 * kMaxBatch;
    sr.path = c->io_res + 3 * kMaxBatch;
    sr.path_stride = res->path_stride;
    sr.logits = res->logits ? c->logits_ws : nullptr;
    TSS_TRY(verify_impl(c, &sub, kv, &sr, s, nullptr, orig.data()));
    // results back to the caller's request positions
    int r = 0;
    for (size_t j = 0; j < orig.size(); ++j) {
      const int b = orig[j], n = nn[j];
      TSS_CU(cudaMemcpyAsync(res->accept_len + b, sr.accept_len + j, sizeof(int32_t), cudaMemcpyDeviceToDevice, s));
      TSS_CU(cudaMemcpyAsync(res->bonus + b, sr.bonus + j, sizeof(int32_t), cudaMemcpyDeviceToDevice, s));
      TSS_CU(cudaMemcpyAsync(res->new_ctx_len + b, sr.new_ctx_len + j, sizeof(int32_t), cudaMemcpyDeviceToDevice, s));
      TSS_CU(cudaMemcpyAsync(res->path + static_cast<size_t>(b) * res->path_stride,
                             sr.path + j * static_cast<size_t>(res->path_stride), sizeof(int32_t) * res->path_stride,
                             cudaMemcpyDeviceToDevice, s));
      if (res->logits)
        TSS_CU(cudaMemcpyAsync(res->logits + off[b] * V, c->logits_ws + r * V, sizeof(float) * n * V,
                               cudaMemcpyDeviceToDevice, s));
      r += n;
    }
    if (group_events && group_events[g]) TSS_CU(cudaEventRecord(static_cast<cudaEvent_t>(group_events[g]), s));
  }
  if (n_groups) *n_groups = static_cast<int>(keys.size());
  return TSS_OK;
}

tss_status tss_prefill(tss_ctx* c, int n_req, const int32_t* n_tokens, const int32_t* ctx_len,
                       const int32_t* domain_id, const int32_t* kv_slot, const int32_t* tokens, int io_host,
                       const tss_kv_cache* kv, void* stream) {
  if (!c) return fail(TSS_ERR_INVALID_ARG, "ctx is NULL");
  if (n_req < 1 || n_req > c->a.max_batch) return fail(TSS_ERR_INVALID_ARG, "n_req must be in [1, max_batch]");
  if (!n_tokens || !ctx_len || !domain_id || !tokens || !kv)
    return fail(TSS_ERR_INVALID_ARG, "n_tokens, ctx_len, domain_id, tokens and kv are required");
  const cudaStream_t s = static_cast<cudaStream_t>(stream);
  std::vector<long long> off(n_req + 1, 0);
  for (int b = 0; b < n_req; ++b) {
    if (n_tokens[b] < 0 || ctx_len[b] < 0) return fail(TSS_ERR_INVALID_ARG, "n_tokens and ctx_len must be >= 0");
    if (static_cast<long long>(ctx_len[b]) + n_tokens[b] > kv->cap)
      return fail(TSS_ERR_KV_CAPACITY, "ctx_len + n_tokens exceeds KV capacity");
    if (static_cast<long long>(ctx_len[b]) + n_tokens[b] > c->a.max_positions)
      return fail(TSS_ERR_INVALID_ARG, "position beyond max_positions");
    off[b + 1] = off[b] + n_tokens[b];
  }
  if (c->pf_enabled && c->D == 128 && c->d % 8 == 0 && c->d <= 256 * 8 * 4) {
    // compute-bound path: the requests of one skip set share passes of up to pf_tmax rows, each
    // request's next chunk starting at a multiple of 128 rows
    for (int l = 0; l < c->L; ++l)
      if (kv->layer[l] && !aligned16(kv->layer[l])) return fail(TSS_ERR_INVALID_ARG, "KV buffers must be 16-byte aligned");
    std::vector<unsigned long long> skip(n_req);
    for (int b = 0; b < n_req; ++b) {
      const int dom = domain_id[b];
      const bool configured = dom >= 0 && dom < c->a.max_domains && c->phi_valid[dom];
      skip[b] = configured ? c->phi[dom] : 0ull;
      for (int l = 0; l < c->L; ++l)
        if (!((skip[b] >> l) & 1ull) && !kv->layer[l]) return fail(TSS_ERR_INVALID_ARG, "KV buffer of an active layer is NULL");
      const int slot = kv_slot ? kv_slot[b] : b;
      if (slot < 0 || slot >= kv->n_slots) return fail(TSS_ERR_INVALID_ARG, "kv_slot out of range");
    }
    TSS_TRY(pf_workspaces(c));
    bool inject = c->inject_timeouts > 0;  // (tss_inject_timeout: the call's first GEMM)
    if (inject) --c->inject_timeouts;
    std::vector<int> done(n_req, 0), pos, slt;
    std::vector<int4> qt;
    std::vector<char> grouped(n_req, 0);
    for (int b0 = 0; b0 < n_req; ++b0) {
      if (grouped[b0]) continue;
      std::vector<int> grp;
      for (int b = b0; b < n_req; ++b)
        if (!grouped[b] && skip[b] == skip[b0]) {
          grouped[b] = 1;
          grp.push_back(b);
        }
      for (;;) {
        int T = 0;
        pos.assign(c->pf_tmax, -1);
        slt.assign(c->pf_tmax, 0);
        qt.clear();
        bool any = false;
        for (int b : grp) {
          const int left = n_tokens[b] - done[b];
          if (left <= 0) continue;
          if (!any) TSS_CU(cudaMemsetAsync(c->pf_tok, 0, sizeof(int) * c->pf_tmax, s));
          const int room = c->pf_tmax - T;
          if (room < 128) break;
          const int len = std::min(left, room);
          const int slot = kv_slot ? kv_slot[b] : b;
          const int p0 = ctx_len[b] + done[b];
          TSS_CU(cudaMemcpyAsync(c->pf_tok + T, tokens + off[b] + done[b], sizeof(int32_t) * len,
                                 io_host ? cudaMemcpyHostToDevice : cudaMemcpyDeviceToDevice, s));
          for (int i = 0; i < len; ++i) {
            pos[T + i] = p0 + i;
            slt[T + i] = slot;
          }
          for (int r = 0; r < len; r += 128) qt.push_back(make_int4(T + r, slot, p0 + r, std::min(128, len - r)));
          done[b] += len;
          T += (len + 127) / 128 * 128;
          any = true;
        }
        if (!any) break;
        // the attention's work items, the most keys first
        std::stable_sort(qt.begin(), qt.end(), [](const int4& a, const int4& b2) { return a.z + a.w > b2.z + b2.w; });
        TSS_CU(cudaMemcpyAsync(c->pf_pos, pos.data(), sizeof(int) * T, cudaMemcpyHostToDevice, s));
        TSS_CU(cudaMemcpyAsync(c->pf_slot, slt.data(), sizeof(int) * T, cudaMemcpyHostToDevice, s));
        TSS_CU(cudaMemcpyAsync(c->pf_qt, qt.data(), sizeof(int4) * qt.size(), cudaMemcpyHostToDevice, s));
        TSS_TRY(pf_pass(c, T, static_cast<int>(qt.size()), skip[b0], kv, s, inject));
        inject = false;
      }
    }
    return TSS_OK;
  }
  // Rounds of verification steps: each request still holding tokens adds a chain of up to
  // max_nodes of them (row 0, the chain's root, is not yet cached, exactly like a draft block's
  // root), within max_rows rows per step; the chains' K/V rows stay where the QKV epilogue wrote
  // them (a chain's compaction moves nothing), and the acceptance outputs go to a scratch buffer.
  std::vector<int> done(n_req, 0);
  std::vector<int32_t> nn, cl, dom, slot, par;
  tss_verify_result res{};
  res.accept_len = c->io_res;
  res.bonus = c->io_res + kMaxBatch;
  res.new_ctx_len = c->io_res + 2 * kMaxBatch;
  res.path = c->io_res + 3 * kMaxBatch;
  res.path_stride = c->a.max_nodes + 1;
  res.logits = nullptr;
  for (;;) {
    nn.clear();
    cl.clear();
    dom.clear();
    slot.clear();
    par.clear();
    int rows = 0;
    for (int b = 0; b < n_req && rows < c->a.max_rows; ++b) {
      const int left = n_tokens[b] - done[b];
      if (left <= 0) continue;
      const int len = std::min(std::min(left, c->a.max_nodes), c->a.max_rows - rows);
      const int32_t* src = tokens + off[b] + done[b];
      TSS_CU(cudaMemcpyAsync(c->io_tokens + rows, src, sizeof(int32_t) * len,
                             io_host ? cudaMemcpyHostToDevice : cudaMemcpyDeviceToDevice, s));
      nn.push_back(len);
      cl.push_back(ctx_len[b] + done[b]);
      dom.push_back(domain_id[b]);
      slot.push_back(kv_slot ? kv_slot[b] : b);
      for (int i = 0; i < len; ++i) par.push_back(i - 1);
      done[b] += len;
      rows += len;
    }
    if (nn.empty()) break;
    tss_verify_batch bt{};
    bt.n_req = static_cast<int>(nn.size());
    bt.n_nodes = nn.data();
    bt.ctx_len = cl.data();
    bt.domain_id = dom.data();
    bt.kv_slot = slot.data();
    bt.parent_idx = par.data();
    bt.positions = nullptr;
    bt.tokens = c->io_tokens;
    bt.mode = TSS_MODE_GREEDY;
    bt.temperature = 1.f;
    bt.io_host = 0;
    TSS_TRY(verify_impl(c, &bt, kv, &res, s, nullptr));
  }
  return TSS_OK;
}

tss_status tss_verify_profiled(tss_ctx* c, const tss_verify_batch* bt, const tss_kv_cache* kv,
                               const tss_verify_result* res, void* stream, tss_kernel_times* times) {
  if (!times) return fail(TSS_ERR_INVALID_ARG, "times is NULL");
  Prof prof;
  tss_status st = verify_impl(c, bt, kv, res, static_cast<cudaStream_t>(stream), &prof);
  if (st == TSS_OK) {
    cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) st = fail(TSS_ERR_CUDA, std::string("cudaStreamSynchronize: ") + cudaGetErrorString(e));
  }
  for (size_t i = 0; st == TSS_OK && i + 1 < prof.ev.size(); i += 2) {
    float ms = 0.f;
    cudaError_t e = cudaEventElapsedTime(&ms, prof.ev[i], prof.ev[i + 1]);
    if (e != cudaSuccess) {
      st = fail(TSS_ERR_CUDA, std::string("cudaEventElapsedTime: ") + cudaGetErrorString(e));
      break;
    }
    const int k = prof.kind[i];
    if (k >= 0 && k < TSS_KERNEL_KINDS) {
      times->ms[k] += ms;
      times->launches[k] += 1;
    }
  }
  for (cudaEvent_t e : prof.ev) cudaEventDestroy(e);
  return st;
}

tss_status tss_sync_status(tss_ctx* c, void* stream) {
  if (!c) return fail(TSS_ERR_INVALID_ARG, "ctx is NULL");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  TSS_CU(cudaMemcpyAsync(c->h_status, c->d_status, sizeof(int), cudaMemcpyDeviceToHost, s));
  TSS_CU(cudaMemsetAsync(c->d_status, 0, sizeof(int), s));
  TSS_CU(cudaStreamSynchronize(s));
  const int v = *c->h_status;
  if (v != 0) return fail(v, std::string("device status: ") + tss_status_string(v));
  return TSS_OK;
}

tss_status tss_philox_uniforms(uint64_t seed, uint64_t offset, int n_req, int n_slots, uint32_t* words, float* uniforms,
                               void* stream) {
  if (n_req < 1 || n_slots < 1 || static_cast<long long>(n_req) * n_slots > (1LL << 28))
    return fail(TSS_ERR_INVALID_ARG, "n_req and n_slots must be positive, n_req * n_slots at most 2^28");
  if (!words && !uniforms) return fail(TSS_ERR_INVALID_ARG, "words and uniforms are both NULL");
  if (words && !aligned16(words)) return fail(TSS_ERR_INVALID_ARG, "words must be 16-byte aligned");
  TSS_CU(launch_philox_fill(seed, offset, n_req, n_slots, words, uniforms, static_cast<cudaStream_t>(stream)));
  return TSS_OK;
}

tss_status tss_inject_timeout(tss_ctx* c, int n_steps) {
  if (!c) return fail(TSS_ERR_INVALID_ARG, "ctx is NULL");
  if (n_steps < 0) return fail(TSS_ERR_INVALID_ARG, "n_steps must be >= 0");
  c->inject_timeouts = n_steps;
  return TSS_OK;
}

tss_status tss_read_trace(tss_ctx* c, unsigned long long* host, size_t capacity, size_t* n_out) {
  if (!c || !n_out) return fail(TSS_ERR_INVALID_ARG, "NULL argument");
  const size_t n = c->trace ? static_cast<size_t>(c->num_sms) * mk_trace_slots() : 0;
  *n_out = n;
  if (!host || n == 0) return TSS_OK;
  if (capacity < n) return fail(TSS_ERR_INVALID_ARG, "trace buffer too small");
  TSS_CU(cudaDeviceSynchronize());
  TSS_CU(cudaMemcpy(host, c->trace, n * sizeof(unsigned long long), cudaMemcpyDeviceToHost));
  return TSS_OK;
}

tss_status tss_linear(tss_ctx* c, const void* x, const void* w, float* y, int m_rows, int k_dim, int n_out, void* stream) {
  if (!c || !x || !w || !y) return fail(TSS_ERR_INVALID_ARG, "NULL argument");
  if (m_rows < 1 || m_rows > kMaxRows || m_rows > c->a.max_rows) return fail(TSS_ERR_INVALID_ARG, "m_rows out of range");
  if (k_dim < 64 || k_dim % 64 != 0) return fail(TSS_ERR_INVALID_ARG, "k_dim must be a positive multiple of 64");
  if (n_out < 128 || n_out % 128 != 0) return fail(TSS_ERR_INVALID_ARG, "n_out must be a positive multiple of 128");
  if (!aligned16(x) || !aligned16(w)) return fail(TSS_ERR_INVALID_ARG, "x and w must be 16-byte aligned");
  const int n_pad = pad_to(m_rows, 16);
  CUtensorMap tx, tw;
  if (!make_tmap(&tx, x, k_dim, m_rows, 1, n_pad, 2) || !make_tmap(&tw, w, k_dim, n_out, 1, 128, 3))
    return fail(TSS_ERR_CUDA, "cuTensorMapEncodeTiled failed");
  GemmParams g = gemm_base(c, n_pad);
  g.slot = -1;
  g.m_raw = m_rows;
  g.layer_fixed = 0;
  g.out = y;
  g.out_ld = n_out;
  g.o_real = n_out;
  g.step = nullptr;
  return run_gemm(c, kEpiStore, tw, tx, g, n_out / 128, k_dim / 64, static_cast<cudaStream_t>(stream), false);
}

}  // extern "C"
