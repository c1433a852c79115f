// Compute-bound prompt prefill under the skip mask (Sec. "Domain-Aware Skip Controller": the
// mask is fixed for the whole request, prompt included; App. "Models": the LLaMA block).
//
// The prompt chunks of requests with the same skip set (each starting at a multiple of 128 rows
// of one pass of up to 4096 rows) run through the layers the skip set keeps, all rows at once: per
// layer RMSNorm, the fused QKV projection with RoPE whose K and V rows are appended to the cache,
// causal attention over the cache, the O projection with the residual, RMSNorm, gate/up with
// SwiGLU and the down projection with the residual.  Nothing past the last layer is computed (the
// prompt's logits are not needed).
//
// GEMMs (pf_gemm_kernel): out[t][o] = sum_k X[t][k] W[o][k] with the weights on the MMA's M side
// (128-row tiles, the pre-tiled 128-byte-swizzled images the verification kernels stream) and
// 128 tokens on the N side; a CTA takes two weight tiles against one token tile at a time (two
// accumulators sharing the token operand) through its whole K loop (no split); items are taken
// weight-pair-major by a persistent grid so that the CTAs working at the same time share weight
// tiles through L2; four groups of epilogue warps keep up with the MMAs.  X is held as two bf16
// parts (hi = bf16(x), lo = bf16(x - hi)), both multiplied by the weights into one fp32
// accumulator in tensor memory, as on the verification path.  Attention (pf_attn_kernel): one CTA
// per (head, 128-query tile of one request), queries on the MMA's M side, 64-key tiles of the
// cache by TMA, S = Q K^T and O += P V in tensor memory, one thread per query row for the online
// softmax; keys past a query's position are masked (causal).
#include "internal.h"

namespace tss {

namespace {

constexpr int kPfThreads = 192;  // attention: warp 0 TMA, warp 1 MMA (+ TMEM), warps 2-5 softmax
constexpr int kPgGroups = 4;     // GEMM epilogue groups of four warps (one per TMEM lane quarter)
constexpr int kPgThreads = 64 + 128 * kPgGroups;  // warp 0 copies, warp 1 MMA (+ TMEM), then the epilogue groups
constexpr int kPfStages = 3;
constexpr uint32_t kPfA = 128 * 64 * 2;      // weight block: 16 KiB
constexpr uint32_t kPfB = 128 * 64 * 2;      // 128 tokens x 64 columns of one part: 16 KiB
constexpr uint32_t kPfStage = 2 * kPfA + 2 * kPfB;  // two weight blocks, the token block's two parts
constexpr uint32_t kPfAccCols = 128;         // one accumulator: 128 token columns

__host__ __device__ inline size_t pf_gemm_smem() {
  return 1024 + static_cast<size_t>(kPfStages) * kPfStage + kPgGroups * 16 * 128 * 4;  // + exchange per group
}

__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

__device__ __forceinline__ void pf_split_store(__nv_bfloat16* hi, __nv_bfloat16* lo, size_t i, float x) {
  const __nv_bfloat16 h = __float2bfloat16_rn(x);
  hi[i] = h;
  lo[i] = __float2bfloat16_rn(x - __bfloat162float(h));
}

}  // namespace

// ---------------------------------------------------------------------------------------------
// Embedding and RMSNorm
// ---------------------------------------------------------------------------------------------
__global__ void pf_embed_kernel(const PfParams p) {
  const int j = blockIdx.x;
  if (j >= p.T) return;
  int tok = p.tokens[j];
  if (tok < 0 || tok >= p.vocab) {
    report(p.status, kStatusCheck);
    tok = 0;
  }
  const __nv_bfloat16* e = p.embed + static_cast<size_t>(tok) * p.d_model;
  for (int c = threadIdx.x; c < p.d_model; c += blockDim.x) p.h[static_cast<size_t>(j) * p.d_model + c] = __bfloat162float(e[c]);
}

// x = h / sqrt(mean(h^2) + eps) * g, as bf16 hi + lo (one block per token row): each thread holds
// kPfNormV groups of 8 consecutive features in registers between the sum of squares and the scaling
// (d_model <= 256 threads x 8 x kPfNormV).
constexpr int kPfNormV = 4;
__global__ void __launch_bounds__(256) pf_norm_kernel(const PfParams p, const float* g) {
  const int j = blockIdx.x;
  if (j >= p.T) return;
  const float* h = p.h + static_cast<size_t>(j) * p.d_model;
  float x[kPfNormV][8];
  float ss = 0.f;
#pragma unroll
  for (int v = 0; v < kPfNormV; ++v) {
    const int c = (v * blockDim.x + threadIdx.x) * 8;
    if (c < p.d_model) {
      const float4 a = *reinterpret_cast<const float4*>(h + c), b = *reinterpret_cast<const float4*>(h + c + 4);
      x[v][0] = a.x; x[v][1] = a.y; x[v][2] = a.z; x[v][3] = a.w;
      x[v][4] = b.x; x[v][5] = b.y; x[v][6] = b.z; x[v][7] = b.w;
#pragma unroll
      for (int i = 0; i < 8; ++i) ss += x[v][i] * x[v][i];
    }
  }
  __shared__ float red[32];
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
  __syncthreads();
  if (threadIdx.x < 32) {
    float v = threadIdx.x < (blockDim.x >> 5) ? red[threadIdx.x] : 0.f;
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (threadIdx.x == 0) red[0] = v;
  }
  __syncthreads();
  const float inv = rsqrtf(red[0] / static_cast<float>(p.d_model) + p.rms_eps);
#pragma unroll
  for (int v = 0; v < kPfNormV; ++v) {
    const int c = (v * blockDim.x + threadIdx.x) * 8;
    if (c < p.d_model) {
      const float4 ga = *reinterpret_cast<const float4*>(g + c), gb = *reinterpret_cast<const float4*>(g + c + 4);
      const float gg[8] = {ga.x, ga.y, ga.z, ga.w, gb.x, gb.y, gb.z, gb.w};
      uint32_t hw[4], lw[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float y0 = x[v][2 * i] * inv * gg[2 * i], y1 = x[v][2 * i + 1] * inv * gg[2 * i + 1];
        hw[i] = pack_bf16(y0, y1);
        lw[i] = pack_bf16(y0 - __uint_as_float(hw[i] << 16), y1 - __uint_as_float(hw[i] & 0xffff0000u));
      }
      const size_t e = static_cast<size_t>(j) * p.x_ld + c;
      *reinterpret_cast<uint4*>(p.xh + e) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
      *reinterpret_cast<uint4*>(p.xl + e) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
    }
  }
}

// ---------------------------------------------------------------------------------------------
// Token-tiled GEMM
// ---------------------------------------------------------------------------------------------
namespace {

// OR of v over the epilogue threads (named barrier 2), which it also synchronises.
__device__ __forceinline__ bool pf_epi_or(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 q, %1, 0;\n\t"
      "bar.red.or.pred p, 2, %2, q;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(r)
      : "r"(v ? 1u : 0u), "n"(128 * kPgGroups)
      : "memory");
  return r != 0;
}

// One 16-token chunk (tokens j0 .. j0 + 15) of output row r of weight tile t; xch: [16][128]
// exchange (the group's own, synchronised by named barrier `bar` of its 128 threads) for the row
// pairs of RoPE (r, r ^ head_dim / 2) and SwiGLU (gate r, up r + 64).
template <int EPI>
__device__ __forceinline__ void pf_epilogue(const PfParams& p, const PfGemm& g, float* xch, int t, int r, int j0,
                                            const float* v, int bar) {
  if constexpr (EPI == kPfEpiResid) {
    const int o = t * 128 + r;
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
      const int j = j0 + jj;
      if (j < p.T) p.h[static_cast<size_t>(j) * p.d_model + o] += v[jj];
    }
  } else if constexpr (EPI == kPfEpiQkv) {
    const int d = p.d_model, D = p.head_dim, half = D >> 1;
    const int o = t * 128 + r;
    const int sec = o / d;  // 0: q, 1: k, 2: v (uniform over the tile: d is a multiple of 128)
    const int f = o - sec * d;
    const int head = f / D, dim = f - head * D;
    float out[16];
    if (sec < 2) {
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) xch[jj * 128 + r] = v[jj];
      named_bar_sync(bar, 128);
      const int pr = r ^ half, i = dim & (half - 1);
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) {
        const int pos = j0 + jj < p.T ? p.row_pos[j0 + jj] : -1;
        out[jj] = 0.f;
        if (pos >= 0) {
          const float c = p.rope_cos[static_cast<size_t>(pos) * half + i];
          const float s = p.rope_sin[static_cast<size_t>(pos) * half + i];
          const float pv = xch[jj * 128 + pr];
          out[jj] = dim < half ? v[jj] * c - pv * s : v[jj] * c + pv * s;
        }
      }
      named_bar_sync(bar, 128);
    } else {
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) out[jj] = v[jj];
    }
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
      const int j = j0 + jj;
      if (j >= p.T) continue;
      const int pos = p.row_pos[j];
      if (pos < 0) continue;  // gap row
      if (sec == 0) {
        pf_split_store(p.qh, p.ql, static_cast<size_t>(j) * d + f, out[jj]);
      } else {
        const size_t row =
            ((static_cast<size_t>(p.row_slot[j]) * 2 + (sec - 1)) * p.n_heads + head) * static_cast<size_t>(p.kv_cap) +
            static_cast<size_t>(pos);
        p.kv[row * D + dim] = __float2bfloat16_rn(out[jj]);
      }
    }
  } else if constexpr (EPI == kPfEpiSwiglu) {
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) xch[jj * 128 + r] = v[jj];
    named_bar_sync(bar, 128);
    if (r < 64) {
      const int fcol = t * 64 + r;
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) {
        const int j = j0 + jj;
        if (j < p.T) {
          const float gt = v[jj], up = xch[jj * 128 + r + 64];
          pf_split_store(p.uh, p.ul, static_cast<size_t>(j) * p.u_ld + fcol, gt / (1.f + expf(-gt)) * up);
        }
      }
    }
    named_bar_sync(bar, 128);
  }
  (void)g;
}

}  // namespace

// Work item = (pair of weight tiles 2w, 2w + 1; token tile u): the two weight tiles share every
// stage's token operand, so a stage of 64 KiB feeds 4 MMAs of 128 x 128 x 16 per k16 step (the
// copy bytes per MMA are half those of one weight tile per item, which L2 bandwidth binds).
template <int EPI>
__global__ void __launch_bounds__(kPgThreads, 1) pf_gemm_kernel(const __grid_constant__ CUtensorMap tm_xh,
                                                                 const __grid_constant__ CUtensorMap tm_xl,
                                                                 const PfParams p, const PfGemm g) {
  extern __shared__ uint8_t pf_dyn[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(pf_dyn) + 1023) & ~uintptr_t(1023));
  float* xch0 = reinterpret_cast<float*>(base + kPfStages * kPfStage);  // [group][16][128]
  __shared__ uint64_t full[kPfStages], empty[kPfStages], acc_full[2], acc_empty[2], drain;
  __shared__ uint32_t tslot;
  __shared__ int abort_s;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int n_u = (p.T + 127) >> 7;         // token tiles
  const int n_w = (g.n_o + 1) >> 1;         // weight-tile pairs (the last may hold one tile)
  const long long n_items = static_cast<long long>(n_w) * n_u;
  if (tid == 0) {
    for (int i = 0; i < kPfStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 4 * kPgGroups);
    }
    mbar_init(&drain, 1);
    abort_s = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&tslot, 4 * kPfAccCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = tslot;
  volatile int* abort = &abort_s;
  const __nv_bfloat16* wl = g.w + static_cast<size_t>(g.layer) * g.w_layer_elems;

  if (warp == 0) {
    // ---------------- producer: both weight blocks and both token parts of each k-block ----------------
    if (lane == 0) {
      prefetch_tmap(&tm_xh);
      prefetch_tmap(&tm_xl);
      long long it = 0;
      bool ok = true;
      for (long long item = blockIdx.x; item < n_items && ok; item += gridDim.x) {
        const int w = static_cast<int>(item / n_u), u = static_cast<int>(item - static_cast<long long>(w) * n_u);
        const int t0 = 2 * w;
        const bool two = t0 + 1 < g.n_o;
        for (int k = 0; k < g.kb; ++k, ++it) {
          const int s = static_cast<int>(it % kPfStages);
          if (it >= kPfStages && !mbar_wait(&empty[s], static_cast<uint32_t>((it / kPfStages) - 1) & 1u, abort, p.status)) {
            ok = false;
            break;
          }
          uint8_t* st = base + s * kPfStage;
          mbar_arrive_expect_tx(&full[s], (two ? 2 : 1) * kPfA + 2 * kPfB);
          bulk_load(st, wl + (static_cast<size_t>(t0) * g.kb + k) * kTileElems, kPfA, &full[s]);
          if (two) bulk_load(st + kPfA, wl + (static_cast<size_t>(t0 + 1) * g.kb + k) * kTileElems, kPfA, &full[s]);
          tma_load_2d(st + 2 * kPfA, &tm_xh, &full[s], k * 64, u * 128);
          tma_load_2d(st + 2 * kPfA + kPfB, &tm_xl, &full[s], k * 64, u * 128);
        }
      }
      for (long long v = it - 1; v >= 0 && v >= it - kPfStages; --v) {
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(&full[v % kPfStages], static_cast<uint32_t>(v / kPfStages) & 1u))
          if (globaltimer_ns() - t0 > kWaitLimitNs) break;
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer: per k16 step, (A0, A1) x (hi, lo) into two accumulators ----------------
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_m128(128);
      long long it = 0;
      int n = 0;
      bool ok = true;
      // fault injection: CTA 0 issues no MMA, so its epilogue's first wait runs out
      const long long n_issue = g.withhold && blockIdx.x == 0 ? 0 : n_items;
      for (long long item = blockIdx.x; item < n_issue && ok; item += gridDim.x, ++n) {
        const int w = static_cast<int>(item / n_u);
        const bool two = 2 * w + 1 < g.n_o;
        const int buf = n & 1;
        if (n >= 2 && !mbar_wait(&acc_empty[buf], static_cast<uint32_t>((n >> 1) - 1) & 1u, abort, p.status)) break;
        tc_fence_after();
        const uint32_t d0 = tm + buf * 2 * kPfAccCols, d1 = d0 + kPfAccCols;
        for (int k = 0; k < g.kb; ++k, ++it) {
          const int s = static_cast<int>(it % kPfStages);
          if (!mbar_wait(&full[s], static_cast<uint32_t>(it / kPfStages) & 1u, abort, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a = smem_u32(base + s * kPfStage), b = a + 2 * kPfA;
#pragma unroll
          for (int k16 = 0; k16 < 4; ++k16) {
            const uint64_t bh = sdesc_sw128(b + k16 * 32), bl = sdesc_sw128(b + kPfB + k16 * 32);
            const uint64_t a0 = sdesc_sw128(a + k16 * 32);
            umma_bf16(d0, a0, bh, idesc, (k | k16) ? 1u : 0u);
            umma_bf16(d0, a0, bl, idesc, 1u);
            if (two) {
              const uint64_t a1 = sdesc_sw128(a + kPfA + k16 * 32);
              umma_bf16(d1, a1, bh, idesc, (k | k16) ? 1u : 0u);
              umma_bf16(d1, a1, bl, idesc, 1u);
            }
          }
          umma_commit(&empty[s]);
        }
        if (ok) umma_commit(&acc_full[buf]);
      }
      // every MMA issued has completed before the kernel returns
      umma_commit(&drain);
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&drain, 0))
        if (globaltimer_ns() - t0 > kWaitLimitNs) break;
    }
  } else {
    // ---------------- epilogue warps: TMEM lane quarter = warp & 3, thread r = weight row; group
    // (warp - 2) / 4 takes its share of the 8 token chunks of each accumulator ----------------
    constexpr int kCh = 8 / kPgGroups;
    const int q = warp & 3, r = q * 32 + lane, grp = (warp - 2) >> 2;
    float* xch = xch0 + grp * 16 * 128;
    const int bar = grp == 0 ? 1 : 2 + grp;  // (2 is the vote barrier)
    int n = 0;
    for (long long item = blockIdx.x; item < n_items; item += gridDim.x, ++n) {
      const int w = static_cast<int>(item / n_u), u = static_cast<int>(item - static_cast<long long>(w) * n_u);
      const int buf = n & 1;
      const bool ok = mbar_wait(&acc_full[buf], static_cast<uint32_t>(n >> 1) & 1u, abort, p.status);
      if (pf_epi_or(!ok)) break;
      tc_fence_after();
      for (int a = 0; a < 2; ++a) {
        const int t = 2 * w + a;
        if (t >= g.n_o) break;
        const uint32_t tb = tm + (static_cast<uint32_t>(q * 32) << 16) + (buf * 2 + a) * kPfAccCols;
        for (int ch = kCh * grp; ch < kCh * grp + kCh; ++ch) {
          float v[16];
          tmem_ld16(tb + ch * 16, v);
          pf_epilogue<EPI>(p, g, xch, t, r, u * 128 + ch * 16, v, bar);
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[buf]);
    }
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tm, 4 * kPfAccCols);
  }
}

// ---------------------------------------------------------------------------------------------
// Causal attention of the chunk's queries (head_dim 128)
// ---------------------------------------------------------------------------------------------
namespace {

constexpr int kPaKeys = 64;                          // keys per tile
constexpr int kPaSlots = 3;                          // slots of the K and of the V ring
constexpr uint32_t kPaQPart = 2 * 128 * 128;         // 128 queries x 128 dims bf16: 32 KiB
constexpr uint32_t kPaKV = 2 * kPaKeys * 128;        // 64 keys x 128 dims: 16 KiB (two 8 KiB boxes)
constexpr uint32_t kPaPPart = 128 * kPaKeys * 2;     // 128 queries x 64 keys: 16 KiB
constexpr uint32_t kPaTmem = 256;                    // S x 2 (64 cols each), O (128 cols)

__host__ __device__ inline size_t pf_attn_smem() {
  return 1024 + 2 * kPaQPart + 2 * kPaSlots * kPaKV + 2 * 2 * kPaPPart;
}

__device__ __forceinline__ uint64_t pa_desc_mn(uint32_t saddr, uint32_t lbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>(1024 >> 4) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}

__device__ __forceinline__ void pa_st16(uint32_t taddr, const float* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16};" ::"r"(taddr),
      "f"(v[0]), "f"(v[1]), "f"(v[2]), "f"(v[3]), "f"(v[4]), "f"(v[5]), "f"(v[6]), "f"(v[7]), "f"(v[8]), "f"(v[9]),
      "f"(v[10]), "f"(v[11]), "f"(v[12]), "f"(v[13]), "f"(v[14]), "f"(v[15])
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// OR of v over the 128 softmax threads (named barrier 1), which it also synchronises.
__device__ __forceinline__ bool pa_or(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 q, %1, 0;\n\t"
      "bar.red.or.pred p, 1, 128, q;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(r)
      : "r"(v ? 1u : 0u)
      : "memory");
  return r != 0;
}

}  // namespace

// Grid (heads, query tiles of p.qtiles, which the host orders heaviest first, so that the CTAs
// with the most keys start first); the KV map has 64-row boxes; tm_q: q hi / lo maps over
// [T_max][d].
__global__ void __launch_bounds__(kPfThreads, 1) pf_attn_kernel(const __grid_constant__ CUtensorMap tm_qh,
                                                                const __grid_constant__ CUtensorMap tm_ql,
                                                                const __grid_constant__ CUtensorMap tm_kv,
                                                                const PfParams p) {
  extern __shared__ uint8_t pa_dyn[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(pa_dyn) + 1023) & ~uintptr_t(1023));
  uint8_t* sq = base;                                // Q hi (2 boxes), Q lo (2 boxes)
  uint8_t* sk = sq + 2 * kPaQPart;                   // [slot] K
  uint8_t* sv = sk + kPaSlots * kPaKV;               // [slot] V
  uint8_t* sp = sv + kPaSlots * kPaKV;               // [2] P hi, P lo
  __shared__ uint64_t qfull, kfull[kPaSlots], kempty[kPaSlots], vfull[kPaSlots], vempty[kPaSlots];
  __shared__ uint64_t s_full[2], s_free[2], p_full[2], p_free[2], o_full, drain;
  __shared__ uint32_t tslot;
  __shared__ int abort_s;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int h = blockIdx.x;
  const int4 qi = p.qtiles[blockIdx.y];  // (first row, slot, position of the first row, rows)
  const int H = p.n_heads, D = 128;
  const int q0 = qi.x, slot = qi.y, pos_t0 = qi.z, nrow = qi.w;
  const int key_end = pos_t0 + nrow;  // keys any query of the tile may see
  const int n = (key_end + kPaKeys - 1) / kPaKeys;
  if (tid == 0) {
    mbar_init(&qfull, 1);
    for (int i = 0; i < kPaSlots; ++i) {
      mbar_init(&kfull[i], 1);
      mbar_init(&kempty[i], 1);
      mbar_init(&vfull[i], 1);
      mbar_init(&vempty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&s_free[i], 4);
      mbar_init(&p_full[i], 1);
      mbar_init(&p_free[i], 1);
    }
    mbar_init(&o_full, 1);
    mbar_init(&drain, 1);
    abort_s = 0;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&tslot, kPaTmem);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = tslot;
  volatile int* abort = &abort_s;
  const size_t cap = static_cast<size_t>(p.kv_cap);
  const int rowK = static_cast<int>(((static_cast<size_t>(slot) * 2) * H + h) * cap);
  const int rowV = rowK + static_cast<int>(static_cast<size_t>(H) * cap);

  if (warp == 0) {
    // ---------------- TMA producer: Q once, then K and V of every key tile ----------------
    if (lane == 0) {
      prefetch_tmap(&tm_kv);
      mbar_arrive_expect_tx(&qfull, 2 * kPaQPart);
      tma_load_2d(sq, &tm_qh, &qfull, h * D, q0);
      tma_load_2d(sq + kPaQPart / 2, &tm_qh, &qfull, h * D + 64, q0);
      tma_load_2d(sq + kPaQPart, &tm_ql, &qfull, h * D, q0);
      tma_load_2d(sq + kPaQPart + kPaQPart / 2, &tm_ql, &qfull, h * D + 64, q0);
      int nk = 0, nv = 0;
      for (int t = 0; t < n; ++t) {
        const int s = t % kPaSlots;
        if (t >= kPaSlots && !mbar_wait(&kempty[s], ((t / kPaSlots) - 1) & 1, abort, p.status)) break;
        mbar_arrive_expect_tx(&kfull[s], kPaKV);
        tma_load_2d(sk + s * kPaKV, &tm_kv, &kfull[s], 0, rowK + t * kPaKeys);
        tma_load_2d(sk + s * kPaKV + kPaKV / 2, &tm_kv, &kfull[s], 64, rowK + t * kPaKeys);
        ++nk;
        if (t >= kPaSlots && !mbar_wait(&vempty[s], ((t / kPaSlots) - 1) & 1, abort, p.status)) break;
        mbar_arrive_expect_tx(&vfull[s], kPaKV);
        tma_load_2d(sv + s * kPaKV, &tm_kv, &vfull[s], 0, rowV + t * kPaKeys);
        tma_load_2d(sv + s * kPaKV + kPaKV / 2, &tm_kv, &vfull[s], 64, rowV + t * kPaKeys);
        ++nv;
      }
      auto drain_bar = [](uint64_t* bar, uint32_t parity) {
        const uint64_t t0 = globaltimer_ns();
        while (!mbar_try_wait(bar, parity))
          if (globaltimer_ns() - t0 > kWaitLimitNs) return;
      };
      drain_bar(&qfull, 0);
      for (int u = nk - 1; u >= 0 && u >= nk - kPaSlots; --u) drain_bar(&kfull[u % kPaSlots], (u / kPaSlots) & 1);
      for (int u = nv - 1; u >= 0 && u >= nv - kPaSlots; --u) drain_bar(&vfull[u % kPaSlots], (u / kPaSlots) & 1);
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer: S(t) = Q K^T, then O += P(t - 1) V ----------------
    if (lane == 0) {
      const uint32_t idS = idesc_bf16_m128(kPaKeys), idPV = idesc_bf16_m128(D) | (1u << 16);  // (B MN-major)
      const uint32_t q_a = smem_u32(sq), k_a = smem_u32(sk), v_a = smem_u32(sv), p_a = smem_u32(sp);
      bool ok = mbar_wait(&qfull, 0, abort, p.status);
      for (int t = 0; ok && t <= n; ++t) {
        if (t < n) {
          const int s = t % kPaSlots;
          if (!mbar_wait(&kfull[s], (t / kPaSlots) & 1, abort, p.status)) break;
          if (t >= 2 && !mbar_wait(&s_free[t & 1], ((t >> 1) - 1) & 1, abort, p.status)) break;
          tc_fence_after();
          const uint32_t dS = tm + (t & 1) * kPaKeys;
#pragma unroll
          for (int part = 0; part < 2; ++part)
#pragma unroll
            for (int kb = 0; kb < 2; ++kb)
#pragma unroll
              for (int k16 = 0; k16 < 4; ++k16)
                umma_bf16(dS, sdesc_sw128(q_a + part * kPaQPart + kb * (kPaQPart / 2) + k16 * 32),
                          sdesc_sw128(k_a + s * kPaKV + kb * (kPaKV / 2) + k16 * 32), idS, (part | kb | k16) ? 1u : 0u);
          umma_commit(&s_full[t & 1]);
          umma_commit(&kempty[s]);
        }
        if (t >= 1) {
          const int u = t - 1, s = u % kPaSlots;
          if (!mbar_wait(&vfull[s], (u / kPaSlots) & 1, abort, p.status)) break;
          if (!mbar_wait(&p_full[u & 1], (u >> 1) & 1, abort, p.status)) break;
          tc_fence_after();
          const uint32_t pb = p_a + (u & 1) * 2 * kPaPPart;
#pragma unroll
          for (int part = 0; part < 2; ++part)
#pragma unroll
            for (int kk = 0; kk < kPaKeys / 16; ++kk)
              umma_bf16(tm + 128, sdesc_sw128(pb + part * kPaPPart + kk * 32),
                        pa_desc_mn(v_a + s * kPaKV + kk * 16 * 128, kPaKV / 2), idPV, (u | part | kk) ? 1u : 0u);
          umma_commit(&vempty[s]);
          umma_commit(&p_free[u & 1]);
          if (u == n - 1) umma_commit(&o_full);
        }
      }
      umma_commit(&drain);
      const uint64_t t0 = globaltimer_ns();
      while (!mbar_try_wait(&drain, 0))
        if (globaltimer_ns() - t0 > kWaitLimitNs) break;
    }
  } else {
    // ---------------- softmax: thread = query row (TMEM lane) ----------------
    const int qg = warp & 3, qr = qg * 32 + lane, st = tid - 64;
    const uint32_t lanes = static_cast<uint32_t>(qg * 32) << 16;
    const int j = q0 + qr;                  // row of this query
    const bool valid = qr < nrow;
    const int pq = pos_t0 + qr;             // its position: keys <= pq are visible
    const float scale = 1.4426950408889634f / sqrtf(static_cast<float>(D));
    float m = -INFINITY, l = 0.f;
    bool ok = true;
    for (int t = 0; t < n; ++t) {
      ok = mbar_wait(&s_full[t & 1], (t >> 1) & 1, abort, p.status);
      if (pa_or(!ok)) break;
      tc_fence_after();
      float s[kPaKeys];
#pragma unroll
      for (int c = 0; c < kPaKeys / 16; ++c) tmem_ld16(tm + lanes + (t & 1) * kPaKeys + c * 16, s + c * 16);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_free[t & 1]);
      float mt = -INFINITY;
#pragma unroll
      for (int c = 0; c < kPaKeys; ++c) {
        const int key = t * kPaKeys + c;
        s[c] = (valid && key <= pq) ? s[c] * scale : -INFINITY;
        mt = fmaxf(mt, s[c]);
      }
      // the row's running max is raised only when the tile exceeds it by more than 2^8; the
      // warp rescales its rows of O together (tensor-memory access is warp-wide)
      const bool raise = mt > m + 8.f;
      float alpha = 1.f;
      if (raise) {
        alpha = m == -INFINITY ? 1.f : exp2f(m - mt);
        m = mt;
        l *= alpha;
      }
      ok = t < 2 || mbar_wait(&p_free[t & 1], ((t >> 1) - 1) & 1, abort, p.status);
      if (t >= 1 && __any_sync(0xffffffffu, raise && alpha != 1.f) && ok)
        ok = mbar_wait(&p_free[(t - 1) & 1], ((t - 1) >> 1) & 1, abort, p.status);
      // in the last tile, the V rows past the keys (stale or unwritten cache rows) are zeroed
      if (ok && t == n - 1) {
        const int s_ = t % kPaSlots, r0 = key_end - t * kPaKeys;
        ok = mbar_wait(&vfull[s_], (t / kPaSlots) & 1, abort, p.status);
        if (ok && st >= r0 && st < kPaKeys) {
          uint4* v0 = reinterpret_cast<uint4*>(sv + s_ * kPaKV + st * 128);
          uint4* v1 = reinterpret_cast<uint4*>(sv + s_ * kPaKV + kPaKV / 2 + st * 128);
#pragma unroll
          for (int i = 0; i < 8; ++i) v0[i] = v1[i] = make_uint4(0, 0, 0, 0);
        }
      }
      if (pa_or(!ok)) break;
      if (t >= 1 && __any_sync(0xffffffffu, raise && alpha != 1.f)) {
        tc_fence_after();
        float o[16];
#pragma unroll
        for (int c = 0; c < D / 16; ++c) {
          tmem_ld16(tm + lanes + 128 + c * 16, o);
#pragma unroll
          for (int i = 0; i < 16; ++i) o[i] *= alpha;
          pa_st16(tm + lanes + 128 + c * 16, o);
        }
        tc_fence_before();
      }
      // weights 2^(s - m) as bf16 hi + lo into the P operand (row qr, 64 keys = one 128-byte row)
      const float mb = m == -INFINITY ? 0.f : m;
      uint8_t* ph = sp + (t & 1) * 2 * kPaPPart + qr * 128;
      uint8_t* pl = ph + kPaPPart;
#pragma unroll
      for (int c8 = 0; c8 < kPaKeys / 8; ++c8) {
        uint32_t hw[4], lw[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float w0 = exp2f(s[c8 * 8 + 2 * i] - mb), w1 = exp2f(s[c8 * 8 + 2 * i + 1] - mb);
          l += w0 + w1;
          hw[i] = pack_bf16(w0, w1);
          const float h0 = __uint_as_float(hw[i] << 16), h1 = __uint_as_float(hw[i] & 0xffff0000u);
          lw[i] = pack_bf16(w0 - h0, w1 - h1);
        }
        const int sw = (c8 ^ (qr & 7)) << 4;
        *reinterpret_cast<uint4*>(ph + sw) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
        *reinterpret_cast<uint4*>(pl + sw) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
      }
      fence_async_smem();
      named_bar_sync(1, 128);
      if (st == 0) mbar_arrive(&p_full[t & 1]);
    }
    if (ok) {
      ok = mbar_wait(&o_full, 0, abort, p.status);
      if (!pa_or(!ok)) {
        tc_fence_after();
        const float inv = l > 0.f ? 1.f / l : 0.f;
        if (valid && !(l > 0.f)) report(p.status, kStatusCheck);
#pragma unroll
        for (int c = 0; c < D / 16; ++c) {
          float o[16];
          tmem_ld16(tm + lanes + 128 + c * 16, o);
          if (valid) {
            // this row's 16 outputs as bf16 hi and lo parts: two 16-byte stores per part
            uint32_t hw[8], lw[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
              const float x0 = o[2 * i] * inv, x1 = o[2 * i + 1] * inv;
              hw[i] = pack_bf16(x0, x1);
              lw[i] = pack_bf16(x0 - __uint_as_float(hw[i] << 16), x1 - __uint_as_float(hw[i] & 0xffff0000u));
            }
            const size_t e = static_cast<size_t>(j) * p.d_model + h * D + c * 16;
            uint4* ph = reinterpret_cast<uint4*>(p.ah + e);
            uint4* pl = reinterpret_cast<uint4*>(p.al + e);
            ph[0] = make_uint4(hw[0], hw[1], hw[2], hw[3]);
            ph[1] = make_uint4(hw[4], hw[5], hw[6], hw[7]);
            pl[0] = make_uint4(lw[0], lw[1], lw[2], lw[3]);
            pl[1] = make_uint4(lw[4], lw[5], lw[6], lw[7]);
          }
        }
        tc_fence_before();
      }
    }
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tm, kPaTmem);
  }
}

// ---------------------------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------------------------
cudaError_t pf_prepare() {
  cudaError_t e = cudaFuncSetAttribute(pf_gemm_kernel<kPfEpiQkv>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(pf_gemm_smem()));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(pf_gemm_kernel<kPfEpiResid>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(pf_gemm_smem()));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(pf_gemm_kernel<kPfEpiSwiglu>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(pf_gemm_smem()));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(pf_attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(pf_attn_smem()));
  return e;
}

cudaError_t launch_pf_embed(const PfParams& p, cudaStream_t s) {
  return launch_k(pf_embed_kernel, dim3(p.T), dim3(256), 0, s, false, p);
}

cudaError_t launch_pf_norm(const PfParams& p, const float* g, cudaStream_t s) {
  return launch_k(pf_norm_kernel, dim3(p.T), dim3(256), 0, s, false, p, g);
}

cudaError_t launch_pf_gemm(int epi, const CUtensorMap& xh, const CUtensorMap& xl, const PfParams& p, const PfGemm& g,
                           int grid, cudaStream_t s) {
  const long long tiles = static_cast<long long>((g.n_o + 1) / 2) * ((p.T + 127) / 128);
  const dim3 gr(static_cast<unsigned>(tiles < grid ? tiles : grid)), blk(kPgThreads);
  switch (epi) {
    case kPfEpiQkv: return launch_k(pf_gemm_kernel<kPfEpiQkv>, gr, blk, pf_gemm_smem(), s, false, xh, xl, p, g);
    case kPfEpiResid: return launch_k(pf_gemm_kernel<kPfEpiResid>, gr, blk, pf_gemm_smem(), s, false, xh, xl, p, g);
    case kPfEpiSwiglu: return launch_k(pf_gemm_kernel<kPfEpiSwiglu>, gr, blk, pf_gemm_smem(), s, false, xh, xl, p, g);
    default: return cudaErrorInvalidValue;
  }
}

cudaError_t launch_pf_attn(const CUtensorMap& qh, const CUtensorMap& ql, const CUtensorMap& kv, const PfParams& p,
                           cudaStream_t s) {
  const dim3 gr(p.n_heads, p.n_qtiles), blk(kPfThreads);
  return launch_k(pf_attn_kernel, gr, blk, pf_attn_smem(), s, false, qh, ql, kv, p);
}

}  // namespace tss
