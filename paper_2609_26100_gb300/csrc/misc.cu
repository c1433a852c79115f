// Row-wise and per-request kernels of the verification step: the skip controller, embedding
// gather, RMSNorm, acceptance (greedy walk or speculative sampling) and KV compaction.
#include "internal.h"

namespace tss {

// ------------------------------------------------------------------------------------------
// Skip controller (Sec. "Domain-Aware Skip Controller", first equation; Sec.
// "Domain-to-Configuration Mapping"): S(x) = Phi(d(x)) if the domain is configured, else the
// empty set -- looked up on the host when the step is enqueued and passed in the step
// descriptor.  From the requests' skip sets it builds, on the device, the ascending list of
// layers that at least one request runs (the only layers that get launches) and, per layer, the
// compacted list of rows of the requests that run it.
// ------------------------------------------------------------------------------------------
__device__ void controller_body(const MiscParams& p) {
  const StepDesc* st = p.step;
  PlanDev* pl = p.plan;
  __shared__ unsigned long long smask[kMaxBatch];
  __shared__ int sact[kMaxLayers];
  __shared__ int s_n;
  const int B = st->B, L = p.n_layers;
  for (int b = threadIdx.x; b < B; b += blockDim.x) {
    const unsigned long long m = st->req_phi[b];
    smask[b] = m;
    pl->req_mask[b] = m;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int n = 0;
    for (int l = 0; l < L; ++l) {
      bool any = false;
      for (int b = 0; b < B; ++b) any = any || !((smask[b] >> l) & 1ull);
      if (any) sact[n++] = l;
    }
    s_n = n;
    pl->n_act = n;
    for (int j = 0; j < n; ++j) pl->act_layer[j] = sact[j];
    if (n != st->n_act_host) report(p.status, kStatusCheck);
  }
  __syncthreads();
  for (int j = threadIdx.x; j <= s_n; j += blockDim.x) {
    const bool final_slot = j == s_n;
    const int slot = final_slot ? kFinalSlot : j;
    const int l = final_slot ? -1 : sact[j];
    int crow = 0;
    for (int b = 0; b < B; ++b) {
      const bool runs = final_slot || !((smask[b] >> l) & 1ull);
      if (runs) {
        pl->slot_crow[slot][b] = crow;
        const int n = st->req_nodes[b], r0 = st->req_rowoff[b];
        for (int i = 0; i < n; ++i) pl->slot_rows[slot][crow + i] = r0 + i;
        crow += n;
      } else {
        pl->slot_crow[slot][b] = -1;
      }
    }
    pl->slot_M[slot] = crow;
  }
}

__global__ void controller_kernel(const MiscParams p) {
  griddep_wait();
  griddep_launch();
  controller_body(p);
}

// h[m] = E[token[m]] (fp32 residual stream).
__global__ void embed_kernel(const MiscParams p) {
  griddep_wait();
  griddep_launch();
  const StepDesc* st = p.step;
  const int m = blockIdx.x;
  if (m >= st->M) return;
  int tok = st->tokens[m];
  if (tok < 0 || tok >= p.vocab) {
    if (threadIdx.x == 0) report(p.status, kStatusCheck);
    tok = 0;
  }
  const __nv_bfloat16* e = p.embed + static_cast<size_t>(tok) * p.d_model;
  float* h = p.h + static_cast<size_t>(m) * p.d_model;
  for (int i = threadIdx.x; i < p.d_model; i += blockDim.x) h[i] = __bfloat162float(e[i]);
}

__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  if (lane == 0) red[w] = v;
  __syncthreads();
  float t = 0.f;
  for (int i = 0; i < nw; ++i) t += red[i];
  __syncthreads();
  return t;
}

// xn[n] = bf16(h[row_n] / sqrt(mean(h^2) + eps) * g) for the compacted rows n of a slot.
__global__ void rmsnorm_kernel(const MiscParams p, int slot, int which) {
  griddep_wait();
  griddep_launch();
  __shared__ float red[32];
  const PlanDev* pl = p.plan;
  const int n = blockIdx.x;
  const bool final_slot = which == 2;
  const int sl = final_slot ? kFinalSlot : slot;
  if (!final_slot && slot >= pl->n_act) return;
  if (n >= pl->slot_M[sl]) return;
  const int m = pl->slot_rows[sl][n];
  const int d = p.d_model;
  const float* g = final_slot ? p.g_final : (which == 0 ? p.g_attn : p.g_mlp) + static_cast<size_t>(pl->act_layer[slot]) * d;
  const float* h = p.h + static_cast<size_t>(m) * d;
  float ss = 0.f;
  for (int i = threadIdx.x; i < d; i += blockDim.x) ss += h[i] * h[i];
  ss = block_sum(ss, red);
  const float rs = rsqrtf(ss / static_cast<float>(d) + p.rms_eps);
  __nv_bfloat16* x = p.xn + static_cast<size_t>(n) * d;
  for (int i = threadIdx.x; i < d; i += blockDim.x) x[i] = __float2bfloat16_rn(h[i] * rs * g[i]);
}

// ------------------------------------------------------------------------------------------
// Acceptance.  Greedy (temperature 0, Sec. "Evaluation Protocol"): from the root, step to the
// lowest-index child whose token equals the argmax of the current row while one exists; the
// bonus is the argmax of the last row reached.  Argmax ties go to the lowest token id.
// ------------------------------------------------------------------------------------------
// Request b's results, written by every thread of the block (a, bonus and path[0..a] are the
// same in all of them; path is in shared memory).  The descriptor's fields are read once into
// registers: read inside a loop of stores through the descriptor's pointers, each would be
// reloaded from L2 after every store.
__device__ void write_result(const MiscParams& p, int b, int a, int bonus, const int* path) {
  const StepDesc* st = p.step;
  PlanDev* pl = p.plan;
  const int stride = st->path_stride;
  int* out = st->path + static_cast<size_t>(b) * stride;
  for (int i = threadIdx.x; i < stride; i += blockDim.x) out[i] = i <= a ? path[i] : -1;
  for (int i = threadIdx.x; i <= a; i += blockDim.x) pl->res_path[b][i] = path[i];
  if (threadIdx.x == 0) {
    const int ctx = st->req_ctx[b];
    int* accept_len = st->accept_len;
    int* bonus_out = st->bonus;
    int* new_ctx = st->new_ctx;
    accept_len[b] = a;
    bonus_out[b] = bonus;
    new_ctx[b] = ctx + 1 + a;
    pl->res_accept[b] = a;
  }
}

// Greedy acceptance of request b; returns the accept length (the same in every thread) and
// leaves the accepted path in path[0..a].
__device__ int accept_greedy_body(const MiscParams& p, int b, int* path) {
  const StepDesc* st = p.step;
  __shared__ int am[kMaxNodes];
  __shared__ int s_par[kMaxNodes], s_tok[kMaxNodes];
  __shared__ int s_a, s_bonus;
  const int N = st->req_nodes[b], off = st->req_rowoff[b];
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    s_par[i] = st->row_parent[off + i];
    s_tok[i] = st->tokens[off + i];
  }
  // Argmax of every row over the vocabulary tiles' partials (laid out [tile][row]): thread
  // (g, r), g < G = blockDim / RP, scans row r's tiles g, g + G, ..., so that a warp's loads
  // cover consecutive rows of one tile; then the G results of each row are combined.  The
  // maximum with ties to the lowest token id does not depend on the order of the comparisons.
  auto better = [](float v, int ix, float& bv, int& bi) {
    if (v > bv || (v == bv && ix < bi)) {
      bv = v;
      bi = ix;
    }
  };
  const int RP = N > 32 ? (N + 31) & ~31 : 32, G = blockDim.x / RP;
  const int r = threadIdx.x % RP, g = threadIdx.x / RP, n_vt = p.n_vtiles;
  float bv = -INFINITY;
  int bi = 0x7fffffff;
  if (g < G && r < N) {
    const float* pv = p.amax_val + off + r;
    const int* pi = p.amax_idx + off + r;
    constexpr int kPer = 8;  // tiles per thread in one round of loads
    for (int t0 = g; t0 < n_vt; t0 += kPer * G) {
      float vv[kPer];
      int vi[kPer];
#pragma unroll
      for (int q = 0; q < kPer; ++q) {
        const int t = t0 + q * G;
        const bool in = t < n_vt;
        vv[q] = in ? pv[static_cast<size_t>(t) * kMaxRows] : -INFINITY;
        vi[q] = in ? pi[static_cast<size_t>(t) * kMaxRows] : 0x7fffffff;
      }
#pragma unroll
      for (int q = 0; q < kPer; ++q) better(vv[q], vi[q], bv, bi);
    }
  }
  __shared__ float s_bv[1024];
  __shared__ int s_bi[1024];
  s_bv[threadIdx.x] = bv;
  s_bi[threadIdx.x] = bi;
  __syncthreads();
  if (threadIdx.x < N) {
    float v = -INFINITY;
    int ix = 0x7fffffff;
    for (int gg = 0; gg < G; ++gg) better(s_bv[gg * RP + threadIdx.x], s_bi[gg * RP + threadIdx.x], v, ix);
    am[threadIdx.x] = ix;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int cur = 0, a = 0;
    path[0] = 0;
    while (true) {
      const int want = am[cur];
      int nxt = -1;
      for (int c = cur + 1; c < N; ++c) {
        if (s_par[c] == cur && s_tok[c] == want) {
          nxt = c;
          break;
        }
      }
      if (nxt < 0) break;
      cur = nxt;
      path[++a] = cur;
    }
    s_a = a;
    s_bonus = am[cur];
  }
  __syncthreads();
  const int a = s_a;
  write_result(p, b, a, s_bonus, path);
  return a;
}

__global__ void accept_greedy_kernel(const MiscParams p) {
  griddep_wait();
  griddep_launch();
  if (blockIdx.x >= p.step->B) return;
  __shared__ int path[kMaxNodes];
  accept_greedy_body(p, blockIdx.x, path);
}

// Philox4x32-10 (Salmon et al., SC'11): 10 rounds of the 4x32 Philox round with key bumps.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
  }
  return c;
}

// The generator's output for uniform slot `slot` of request b: counter (slot, request, offset lo,
// offset hi), key (seed lo, seed hi); the uniform is (first word >> 8) * 2^-24, exact in fp32.
__device__ __forceinline__ uint4 philox_slot(uint32_t seed_lo, uint32_t seed_hi, uint32_t off_lo, uint32_t off_hi,
                                             int b, int slot) {
  return philox4x32_10(make_uint4(static_cast<uint32_t>(slot), static_cast<uint32_t>(b), off_lo, off_hi), seed_lo,
                       seed_hi);
}
__device__ __forceinline__ float uniform24(uint32_t x) { return static_cast<float>(x >> 8) * (1.f / 16777216.f); }

__device__ __forceinline__ double draw_uniform(const StepDesc* st, int b, int slot) {
  if (st->uniforms) return static_cast<double>(st->uniforms[static_cast<size_t>(b) * st->uniform_stride + slot]);
  return static_cast<double>(
      uniform24(philox_slot(st->seed_lo, st->seed_hi, st->off_lo, st->off_hi, st->req_rng[b], slot).x));
}

// Diagnostic: the generator's words and uniforms for requests [0, n_req) and slots [0, n_slots)
// of one (seed, offset), laid out [request][slot] (the stream the acceptance draws from).
__global__ void philox_fill_kernel(uint32_t seed_lo, uint32_t seed_hi, uint32_t off_lo, uint32_t off_hi, int n_req,
                                   int n_slots, uint4* words, float* unif) {
  const size_t n = static_cast<size_t>(n_req) * n_slots;
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const int b = static_cast<int>(i / n_slots), slot = static_cast<int>(i - static_cast<size_t>(b) * n_slots);
    const uint4 x = philox_slot(seed_lo, seed_hi, off_lo, off_hi, b, slot);
    if (words) words[i] = x;
    if (unif) unif[i] = uniform24(x.x);
  }
}

cudaError_t launch_philox_fill(uint64_t seed, uint64_t offset, int n_req, int n_slots, uint32_t* words, float* unif,
                               cudaStream_t s) {
  const size_t n = static_cast<size_t>(n_req) * n_slots;
  const int blocks = static_cast<int>((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096);
  philox_fill_kernel<<<blocks, 256, 0, s>>>(static_cast<uint32_t>(seed), static_cast<uint32_t>(seed >> 32),
                                            static_cast<uint32_t>(offset), static_cast<uint32_t>(offset >> 32), n_req,
                                            n_slots, reinterpret_cast<uint4*>(words), unif);
  return cudaGetLastError();
}

template <typename T, typename Op>
__device__ __forceinline__ T block_reduce(T v, T* red, Op op) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) v = op(v, __shfl_xor_sync(0xffffffffu, v, off));
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  if (lane == 0) red[w] = v;
  __syncthreads();
  T t = red[0];
  for (int i = 1; i < nw; ++i) t = op(t, red[i]);
  __syncthreads();
  return t;
}

// Inverse CDF over token ids in ascending order: the smallest v whose running sum of w exceeds
// u * sum(w).  Each thread owns a contiguous chunk; chunk sums are scanned in thread order.
// fp32 throughout: the sums over a 32k vocabulary are accurate to ~1e-6 of the mass, far inside
// the 2e-4 band within which a draw counts as consistent, and fp64 is slow on this GPU.
// Loads of the vocabulary passes are issued kLoadBatch at a time (one round trip per batch
// instead of one per element); every sum keeps the element order of a plain loop.
constexpr int kLoadBatch = 16;

template <typename WFn>
__device__ int inverse_cdf_block(int V, float u, WFn w, float* scan) {
  const int nt = blockDim.x, t = threadIdx.x;
  const int C = (V + nt - 1) / nt;
  const int v0 = min(V, t * C), v1 = min(V, v0 + C);
  float local = 0.f;
  for (int b0 = v0; b0 < v1; b0 += kLoadBatch) {
    float x[kLoadBatch];
#pragma unroll
    for (int j = 0; j < kLoadBatch; ++j) x[j] = b0 + j < v1 ? w(b0 + j) : 0.f;
#pragma unroll
    for (int j = 0; j < kLoadBatch; ++j) local += x[j];  // x + 0 == x: the order of a plain loop
  }
  // exclusive scan of the chunk sums in thread order: warp scans, then the warp totals
  const int lane = t & 31, warp = t >> 5, nw = nt >> 5;
  float incl = local;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  __shared__ float wsum[32];
  if (lane == 31) wsum[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    float x = lane < nw ? wsum[lane] : 0.f;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float y = __shfl_up_sync(0xffffffffu, x, o);
      if (lane >= o) x += y;
    }
    if (lane < nw) wsum[lane] = x;  // inclusive totals of warps 0..lane
  }
  __syncthreads();
  const float before = (warp > 0 ? wsum[warp - 1] : 0.f) + (incl - local);
  scan[t] = before;
  if (t == nt - 1) scan[nt] = before + local;
  __syncthreads();
  __shared__ int sel;
  if (t == 0) sel = -1;
  __syncthreads();
  const float total = scan[nt];
  const float target = u * total;
  const float lo = scan[t], hi = (t + 1 < nt) ? scan[t + 1] : total;
  if (local > 0.f && lo <= target && (target < hi || t + 1 == nt || hi >= total)) {
    float run = lo;
    int pick = -1, last_pos = -1;
    for (int v = v0; v < v1; ++v) {
      const float x = w(v);
      if (x > 0.f) last_pos = v;
      run += x;
      if (run > target && x > 0.f) {
        pick = v;
        break;
      }
    }
    if (pick < 0) pick = last_pos;
    atomicCAS(&sel, -1, pick);
  }
  __syncthreads();
  int r = sel;
  if (r < 0) {  // target at or beyond the total: the last token with positive mass
    __shared__ int lastv;
    if (t == 0) lastv = -1;
    __syncthreads();
    for (int v = v1 - 1; v >= v0; --v)
      if (w(v) > 0.f) {
        atomicMax(&lastv, v);
        break;
      }
    __syncthreads();
    r = lastv < 0 ? 0 : lastv;
  }
  __syncthreads();
  return r;
}

// The same inverse CDF over weights staged in shared memory, when the launch gave the block
// enough dynamic shared memory (cdf_stage_bytes): w(v) is computed once per token with coalesced
// loads into a buffer indexed v + v / 32 (the skew puts the 32 consecutive tokens of each
// thread's chunk in 32 different banks), then the chunk sums, scan and walk above read it there.
// Without it each warp-wide load of the chunk pass touches 32 cache lines.
__device__ __forceinline__ unsigned dyn_smem_bytes() {
  unsigned n;
  asm volatile("mov.u32 %0, %%dynamic_smem_size;" : "=r"(n));
  return n;
}

template <typename WFn>
__device__ int inverse_cdf_staged(int V, float u, WFn w, float* scan) {
  extern __shared__ float cdf_stage[];
  const size_t need = cdf_stage_bytes(V);
  if (need == 0 || dyn_smem_bytes() < need) return inverse_cdf_block(V, u, w, scan);
  // kStage weights per thread are computed before any is stored: the stores could alias the
  // generic loads inside w, so a load after a store would wait for it
  constexpr int kStage = 8;
  const int nt = blockDim.x;
  for (int v0 = threadIdx.x; v0 < V; v0 += kStage * nt) {
    float x[kStage];
#pragma unroll
    for (int j = 0; j < kStage; ++j) x[j] = v0 + j * nt < V ? w(v0 + j * nt) : 0.f;
#pragma unroll
    for (int j = 0; j < kStage; ++j) {
      const int v = v0 + j * nt;
      if (v < V) cdf_stage[v + (v >> 5)] = x[j];
    }
  }
  __syncthreads();
  return inverse_cdf_block(V, u, [&](int v) { return cdf_stage[v + (v >> 5)]; }, scan);
}

// Speculative sampling on a chain draft (rule of the speculative-decoding works the paper cites
// as its base methods): p_i = softmax(logits_i / T); accept draft x_i iff r_i * q_i(x_i) <
// p_{i-1}(x_i); at the first rejection draw the bonus from normalise(max(0, p_{i-1} - q_i));
// if every draft is accepted draw it from p_k.  Uniform slots: r_i at i-1, u_i at k+i-1.
__device__ int accept_sample_body(const MiscParams& p, int b, int* path) {
  const StepDesc* st = p.step;
  __shared__ float scan[1025];
  __shared__ float redf[32];
  const int N = st->req_nodes[b], off = st->req_rowoff[b], k = N - 1, V = p.vocab;
  const float invT = st->inv_temperature;
  auto fmx = [](float a, float c) { return a > c ? a : c; };
  auto fsum = [](float a, float c) { return a + c; };
  int a = 0, bonus = 0;
  for (int i = threadIdx.x; i < N; i += blockDim.x) path[i] = i;  // (read after the first barrier)
  for (int i = 1; i <= k + 1; ++i) {
    const float* lg = st->logits + static_cast<size_t>(off + i - 1) * V;
    const int nt = blockDim.x;
    float mx = -INFINITY;
    for (int b0 = threadIdx.x; b0 < V; b0 += kLoadBatch * nt) {
      float x[kLoadBatch];
#pragma unroll
      for (int j = 0; j < kLoadBatch; ++j) x[j] = b0 + j * nt < V ? lg[b0 + j * nt] : -INFINITY;
#pragma unroll
      for (int j = 0; j < kLoadBatch; ++j) mx = fmx(mx, x[j]);
    }
    mx = block_reduce(mx, redf, fmx);
    float z = 0.f;
    for (int b0 = threadIdx.x; b0 < V; b0 += kLoadBatch * nt) {
      float x[kLoadBatch];
#pragma unroll
      for (int j = 0; j < kLoadBatch; ++j) x[j] = b0 + j * nt < V ? lg[b0 + j * nt] : 0.f;
#pragma unroll
      for (int j = 0; j < kLoadBatch; ++j)
        if (b0 + j * nt < V) z += expf((x[j] - mx) * invT);
    }
    z = block_reduce(z, redf, fsum);
    const float invz = 1.f / z;
    auto pr = [&](int v) { return expf((lg[v] - mx) * invT) * invz; };
    if (i <= k) {
      const int x = st->tokens[off + i];
      const float* q = st->draft_probs + static_cast<size_t>(off + i) * V;
      if (x < 0 || x >= V) {
        if (threadIdx.x == 0) report(p.status, kStatusCheck);
        a = i - 1;
        bonus = 0;
        break;
      }
      const float qx = q[x];
      if (!(qx > 0.f) && threadIdx.x == 0) report(p.status, kStatusCheck);
      const float r = static_cast<float>(draw_uniform(st, b, i - 1));
      if (r * qx < pr(x)) continue;  // accept draft i
      const float u = static_cast<float>(draw_uniform(st, b, k + i - 1));
      bonus = inverse_cdf_staged(V, u, [&](int v) {
        const float d = pr(v) - q[v];
        return d > 0.f ? d : 0.f;
      }, scan);
      a = i - 1;
      break;
    }
    const float u = static_cast<float>(draw_uniform(st, b, 2 * k));
    bonus = inverse_cdf_staged(V, u, pr, scan);
    a = k;
  }
  __syncthreads();
  write_result(p, b, a, bonus, path);
  return a;
}

__global__ void __launch_bounds__(1024) accept_sample_kernel(const MiscParams p) {
  griddep_wait();
  griddep_launch();
  if (blockIdx.x >= p.step->B) return;
  __shared__ int path[kMaxNodes];
  accept_sample_body(p, blockIdx.x, path);
}

// ------------------------------------------------------------------------------------------
// Step prologue for the persistent verify kernel: block 0 runs the skip controller; block
// 1 + m embeds row m and writes, per 128-feature tile t, the partial sum of squares
// ssp[t][m] that the RMSNorm of the first active layer needs.
// ------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) prologue_kernel(const MiscParams p, float* ssp, int* zero_ints, int n_zero) {
  griddep_wait();
  griddep_launch();
  if (blockIdx.x == 0) {
    // counters and the abort word of the persistent kernel start every step at zero, even after
    // a step that gave up on a timeout
    for (int i = threadIdx.x; i < n_zero; i += blockDim.x) zero_ints[i] = 0;
    controller_body(p);
    return;
  }
  const StepDesc* st = p.step;
  const int m = blockIdx.x - 1;
  if (m >= st->M) return;
  int tok = st->tokens[m];
  if (tok < 0 || tok >= p.vocab) {
    if (threadIdx.x == 0) report(p.status, kStatusCheck);
    tok = 0;
  }
  __shared__ float red[16];
  __shared__ unsigned long long smask[kMaxBatch];
  __shared__ int s_l0, s_crow;
  // The first norm phase is the QKV of the union's first layer (or the LM head when every layer
  // is skipped); find this row's compacted position in it, as the controller does.
  for (int b = threadIdx.x; b < st->B; b += blockDim.x) smask[b] = st->req_phi[b];
  __syncthreads();
  if (threadIdx.x == 0) {
    int l0 = -1;
    for (int l = 0; l < p.n_layers && l0 < 0; ++l)
      for (int b = 0; b < st->B; ++b)
        if (!((smask[b] >> l) & 1ull)) {
          l0 = l;
          break;
        }
    const int rb = st->row_req[m];
    int crow = -1;
    if (l0 < 0) {
      crow = m;
    } else if (!((smask[rb] >> l0) & 1ull)) {
      crow = m - st->req_rowoff[rb];
      for (int b = 0; b < rb; ++b)
        if (!((smask[b] >> l0) & 1ull)) crow += st->req_nodes[b];
    }
    s_l0 = l0;
    s_crow = crow;
  }
  __syncthreads();
  const float* gain = s_l0 >= 0 ? p.g_attn + static_cast<size_t>(s_l0) * p.d_model : p.g_final;
  const int xrow = s_crow;
  const __nv_bfloat16* e = p.embed + static_cast<size_t>(tok) * p.d_model;
  float* h = p.h + static_cast<size_t>(m) * p.d_model;
  const int half = threadIdx.x >> 7, r = threadIdx.x & 127;
  const int n_t = p.d_model / 128;
  // every load of the row first (one memory round trip), then the per-tile work
  constexpr int kPer = 32;  // 128-feature tiles per thread half: d_model <= 8192
  float xe[kPer], xg[kPer];
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    const int t = 2 * q + half;
    xe[q] = t < n_t ? __bfloat162float(e[t * 128 + r]) : 0.f;
    xg[q] = t < n_t && xrow >= 0 ? gain[t * 128 + r] : 0.f;
  }
#pragma unroll
  for (int q = 0; q < kPer; ++q) {
    if (2 * q >= n_t) break;
    const int t = 2 * q + half;
    float sq = 0.f;
    if (t < n_t) {
      const float x = xe[q];
      h[t * 128 + r] = x;
      if (xrow >= 0) {
        const float xv = x * xg[q];
        if (p.xs.rows)
          store_split(p.xn, p.xs, xrow, t * 128 + r, xv);
        else
          p.xn[static_cast<size_t>(xrow) * p.d_model + t * 128 + r] = __float2bfloat16_rn(xv);
      }
      sq = x * x;
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, off);
    if ((threadIdx.x & 31) == 0) red[(q & 1) * 8 + (threadIdx.x >> 5)] = sq;
    __syncthreads();  // red is double-buffered by q parity, so one barrier per tile pair
    if (r == 0 && t < n_t)
      ssp[static_cast<size_t>(t) * kMaxRows + m] = (red[(q & 1) * 8 + half * 4] + red[(q & 1) * 8 + half * 4 + 1]) +
                                                   (red[(q & 1) * 8 + half * 4 + 2] + red[(q & 1) * 8 + half * 4 + 3]);
  }
}

// ------------------------------------------------------------------------------------------
// Step finish: acceptance of request b (greedy walk or speculative sampling), then the KV
// compaction of its accepted path in every layer it ran (one 1024-thread block per request).
// ------------------------------------------------------------------------------------------
__global__ void __launch_bounds__(1024) finish_kernel(const MiscParams p) {
  griddep_wait();
  griddep_launch();
  const StepDesc* st = p.step;
  const PlanDev* pl = p.plan;
  const int b = blockIdx.x;
  if (b >= st->B) return;
  __shared__ int path[kMaxNodes];
  const int a = st->mode == TSS_MODE_SAMPLE ? accept_sample_body(p, b, path) : accept_greedy_body(p, b, path);
  if (a <= 0) return;
  // A chain's accepted rows are already in place (path[j] == j): nothing moves in any layer.
  bool moved = false;
  for (int jj = 1; jj <= a; ++jj) moved |= path[jj] != jj;
  if (!moved) return;
  const int D = p.head_dim, H = p.n_heads;
  const size_t cap = static_cast<size_t>(st->kv_cap);
  const size_t ctx = static_cast<size_t>(st->req_ctx[b]);
  const int n_act = pl->n_act;
  // request b's cache region in every layer it ran, looked up by one thread per layer (null
  // where it skipped the layer), so that the copies below wait on no descriptor loads
  __shared__ __nv_bfloat16* s_base[kMaxLayers];
  const size_t slot_off = static_cast<size_t>(st->req_slot[b]) * 2 * H * cap * D;
  for (int j = threadIdx.x; j < n_act; j += blockDim.x)
    s_base[j] = pl->slot_crow[j][b] < 0 ? nullptr : st->kv_layer[pl->act_layer[j]] + slot_off;
  __syncthreads();
  // 16-byte units (head_dim is 64 or 128): unit e = (kind, head, 8 dims) stays with one thread
  // across the path steps, and a later step never reads a row an earlier step wrote, so the
  // in-order copy needs no barrier.
  const int vec = D / 8;
  for (int j = 0; j < n_act; ++j) {
    __nv_bfloat16* base = s_base[j];
    if (!base) continue;
    for (int jj = 1; jj <= a; ++jj) {
      const int src = path[jj];
      if (src == jj) continue;
      for (int e = threadIdx.x; e < 2 * H * vec; e += blockDim.x) {
        const int kind_head = e / vec, u = e - kind_head * vec;
        uint4* row = reinterpret_cast<uint4*>(base + static_cast<size_t>(kind_head) * cap * D);
        row[(ctx + jj) * vec + u] = row[(ctx + src) * vec + u];
      }
    }
  }
}

// ------------------------------------------------------------------------------------------
// KV compaction: for every layer the request ran, cache rows ctx + path[j] move to ctx + j,
// j = 1..a (the root's row stays).  path[j] > j - 1 and increasing, so copying j in increasing
// order never overwrites a row that a later j still reads.  Chains leave the cache unchanged.
// ------------------------------------------------------------------------------------------
__global__ void compact_kernel(const MiscParams p) {
  griddep_wait();
  griddep_launch();
  const StepDesc* st = p.step;
  const PlanDev* pl = p.plan;
  const int head = blockIdx.x, b = blockIdx.y, j = blockIdx.z;
  if (b >= st->B || j >= pl->n_act || pl->slot_crow[j][b] < 0) return;
  const int a = pl->res_accept[b];
  if (a <= 0) return;
  const int D = p.head_dim, H = p.n_heads;
  const size_t cap = static_cast<size_t>(st->kv_cap);
  __nv_bfloat16* K = st->kv_layer[pl->act_layer[j]] + ((static_cast<size_t>(st->req_slot[b]) * 2) * H + head) * cap * D;
  __nv_bfloat16* Vv = K + static_cast<size_t>(H) * cap * D;
  const size_t ctx = static_cast<size_t>(st->req_ctx[b]);
  for (int jj = 1; jj <= a; ++jj) {
    const int src = pl->res_path[b][jj];
    if (src == jj) continue;
    for (int dd = threadIdx.x; dd < D; dd += blockDim.x) {
      K[(ctx + jj) * D + dd] = K[(ctx + src) * D + dd];
      Vv[(ctx + jj) * D + dd] = Vv[(ctx + src) * D + dd];
    }
  }
}

__global__ void bf16_to_f32_kernel(const __nv_bfloat16* src, float* dst, size_t n) {
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n;
       i += static_cast<size_t>(gridDim.x) * blockDim.x)
    dst[i] = __bfloat162float(src[i]);
}

cudaError_t misc_prepare() {
  const int c = cudaSharedmemCarveoutMaxShared;
  const cudaFuncAttribute a = cudaFuncAttributePreferredSharedMemoryCarveout;
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(controller_kernel, a, c)) || (e = cudaFuncSetAttribute(embed_kernel, a, c)) ||
      (e = cudaFuncSetAttribute(rmsnorm_kernel, a, c)) || (e = cudaFuncSetAttribute(accept_greedy_kernel, a, c)) ||
      (e = cudaFuncSetAttribute(accept_sample_kernel, a, c)) || (e = cudaFuncSetAttribute(compact_kernel, a, c)) ||
      (e = cudaFuncSetAttribute(prologue_kernel, a, c)) || (e = cudaFuncSetAttribute(finish_kernel, a, c)))
    return e;
  const int dyn = static_cast<int>(kCdfStageMaxBytes);
  const cudaFuncAttribute mx = cudaFuncAttributeMaxDynamicSharedMemorySize;
  if ((e = cudaFuncSetAttribute(finish_kernel, mx, dyn)) || (e = cudaFuncSetAttribute(accept_sample_kernel, mx, dyn)))
    return e;
  return cudaSuccess;
}

cudaError_t launch_prologue(const MiscParams& p, float* ssp, int* zero_ints, int n_zero, int M, cudaStream_t s,
                            bool pdl) {
  return launch_k(prologue_kernel, dim3(M + 1), dim3(256), 0, s, pdl, p, ssp, zero_ints, n_zero);
}
cudaError_t launch_finish(const MiscParams& p, int B, bool sample, cudaStream_t s, bool pdl) {
  return launch_k(finish_kernel, dim3(B), dim3(1024), sample ? cdf_stage_bytes(p.vocab) : 0, s, pdl, p);
}

cudaError_t launch_controller(const MiscParams& p, cudaStream_t s, bool pdl) {
  return launch_k(controller_kernel, dim3(1), dim3(128), 0, s, pdl, p);
}
cudaError_t launch_embed(const MiscParams& p, int M, cudaStream_t s, bool pdl) {
  return launch_k(embed_kernel, dim3(M), dim3(256), 0, s, pdl, p);
}
cudaError_t launch_rmsnorm(const MiscParams& p, int slot, int which, int M, cudaStream_t s, bool pdl) {
  return launch_k(rmsnorm_kernel, dim3(M), dim3(256), 0, s, pdl, p, slot, which);
}
cudaError_t launch_accept_greedy(const MiscParams& p, int B, cudaStream_t s, bool pdl) {
  return launch_k(accept_greedy_kernel, dim3(B), dim3(256), 0, s, pdl, p);
}
cudaError_t launch_accept_sample(const MiscParams& p, int B, cudaStream_t s, bool pdl) {
  return launch_k(accept_sample_kernel, dim3(B), dim3(1024), cdf_stage_bytes(p.vocab), s, pdl, p);
}
cudaError_t launch_compact(const MiscParams& p, int B, int n_act, cudaStream_t s, bool pdl) {
  if (n_act <= 0) n_act = 1;
  return launch_k(compact_kernel, dim3(p.n_heads, B, n_act), dim3(128), 0, s, pdl, p);
}
// One thread per 16-byte chunk (8 columns) of the source.
__global__ void tile_weights_kernel(const __nv_bfloat16* src, __nv_bfloat16* dst, int rows, int cols) {
  const size_t n_chunks = static_cast<size_t>(rows) * (cols / 8);
  const int kbs = cols / 64;
  for (size_t i = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; i < n_chunks;
       i += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const int row = static_cast<int>(i / (cols / 8));
    const int col = static_cast<int>(i % (cols / 8)) * 8;
    const int t = row >> 7, r = row & 127, kb = col >> 6, c8 = (col & 63) >> 3;
    const size_t blk = static_cast<size_t>(t) * kbs + kb;
    uint8_t* d = reinterpret_cast<uint8_t*>(dst + blk * kTileElems) + r * 128 + ((c8 ^ (r & 7)) << 4);
    *reinterpret_cast<uint4*>(d) = *reinterpret_cast<const uint4*>(src + static_cast<size_t>(row) * cols + col);
  }
}

cudaError_t launch_tile_weights(const __nv_bfloat16* src, __nv_bfloat16* dst, int rows, int cols, cudaStream_t s) {
  const size_t n = static_cast<size_t>(rows) * (cols / 8);
  const int blocks = static_cast<int>(n / 256 + 1 < 16384 ? n / 256 + 1 : 16384);
  tile_weights_kernel<<<blocks, 256, 0, s>>>(src, dst, rows, cols);
  return cudaGetLastError();
}

cudaError_t launch_bf16_to_f32(const __nv_bfloat16* src, float* dst, size_t n, cudaStream_t s) {
  const int blocks = static_cast<int>((n + 255) / 256 < 4096 ? (n + 255) / 256 : 4096);
  bf16_to_f32_kernel<<<blocks > 0 ? blocks : 1, 256, 0, s>>>(src, dst, n);
  return cudaGetLastError();
}

}  // namespace tss
