// Weight-streaming GEMM for the verifier's projections (App. "Models": q/k/v/o projections and the
// SwiGLU MLP of a LLaMA block; the LM head), written for sm_103a.
//
//   D^T[o][n] = sum_k W[o][k] * X[n][k]
//
// The weight matrix is the MMA's M side (128 rows per tile) and the few token rows of a
// verification step (k x batch, padded to a multiple of 16) are the N side, so a 128 x N fp32
// accumulator lives in tensor memory.  Per CTA: one TMA producer thread streams 128x64 weight
// tiles and N x 64 activation tiles (128-byte swizzle) through an mbarrier pipeline, one thread
// issues tcgen05.mma, and four epilogue warps read the accumulator with tcgen05.ld.
//
// Work is split stream-K: the (tile, k-block) iterations are divided evenly over a persistent
// grid, so every SM streams the same number of weight bytes whatever the shape.  A CTA that holds
// only part of a tile writes its partial sum to a scratch slot and bumps the tile's counter; the
// last arrival adds the slots in a fixed order (deterministic) and runs the fused epilogue.
//
// Programmatic dependent launch: the producer issues the first pipeline stages of *weight* tiles
// (which do not depend on the previous kernel) before griddepcontrol.wait, and the activation
// tiles after it, so weight streaming overlaps the previous kernel's tail.
#include <utility>

#include "internal.h"

namespace tss {

constexpr int kGemmThreads = 192;  // warp 0: TMA, warp 1: MMA + TMEM alloc, warps 2-5: epilogue
constexpr uint32_t kWTileBytes = 128 * 64 * 2;

size_t gemm_smem_bytes(int n_pad, int stages) {
  const size_t x_bytes = static_cast<size_t>(n_pad) * 128;
  return 1024                                          // alignment slack
         + static_cast<size_t>(stages) * (kWTileBytes + x_bytes)  // pipeline
         + static_cast<size_t>(2 * stages + 4) * 8      // mbarriers
         + 64                                           // tmem slot, flags
         + 16 * 128 * 4                                 // epilogue exchange tile
         + 2 * 4 * 16 * 4;                              // argmax reduction
}

__device__ __forceinline__ int cta_of(long long i, long long T, int G) {
  return static_cast<int>(((i + 1) * G - 1) / T);
}

__device__ __forceinline__ bool next_segment(long long& it, long long end, int kb, int& t, int& k0, int& k1) {
  if (it >= end) return false;
  t = static_cast<int>(it / kb);
  k0 = static_cast<int>(it - static_cast<long long>(t) * kb);
  const long long tile_end = static_cast<long long>(t + 1) * kb;
  const long long e = end < tile_end ? end : tile_end;
  k1 = static_cast<int>(e - static_cast<long long>(t) * kb);
  it = e;
  return true;
}

struct EpiCtx {
  int M;              // valid token rows
  const int* rows;    // compacted row -> batch row (nullptr: identity)
  int layer;
  float* xch;         // [16][128]
  float* redv;        // [4][16]
  int* redi;          // [4][16]
  int q;              // TMEM lane quarter of this warp
  int lane;
  int et;             // epilogue thread 0..127
};

__device__ __forceinline__ int batch_row(const EpiCtx& e, int j) { return e.rows ? e.rows[j] : j; }

// One 16-column chunk of the accumulator (tokens ch*16 .. ch*16+15) for output row r of tile t.
template <int EPI>
__device__ __forceinline__ void epilogue_chunk(const GemmParams& p, const EpiCtx& e, int t, int r, int ch,
                                               const float* v) {
  const int j0 = ch * 16;
  if constexpr (EPI == kEpiStore) {
    const int o = t * 128 + r;
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
      const int j = j0 + jj;
      if (j < e.M && o < p.o_real) p.out[static_cast<size_t>(j) * p.out_ld + o] = v[jj];
    }
  } else if constexpr (EPI == kEpiResid) {
    const int o = t * 128 + r;
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
      const int j = j0 + jj;
      if (j < e.M) {
        float* hp = p.h + static_cast<size_t>(batch_row(e, j)) * p.d_model + o;
        *hp += v[jj];
      }
    }
  } else if constexpr (EPI == kEpiQkv) {
    const StepDesc* st = p.step;
    const int d = p.d_model, D = p.head_dim, half = D >> 1;
    const int o = t * 128 + r;
    const int sec = o / d;  // 0: q, 1: k, 2: v (uniform over the tile: d is a multiple of 128)
    const int f = o - sec * d;
    const int head = f / D, dim = f - head * D;
    float out[16];
    if (sec < 2) {
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) e.xch[jj * 128 + r] = v[jj];
      named_bar_sync(1, 128);
      const int pr = r ^ half;
      const int i = dim & (half - 1);
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) {
        const int j = j0 + jj;
        out[jj] = 0.f;
        if (j < e.M) {
          const int pos = st->row_pos[batch_row(e, j)];
          const float c = p.rope_cos[static_cast<size_t>(pos) * half + i];
          const float s = p.rope_sin[static_cast<size_t>(pos) * half + i];
          const float pv = e.xch[jj * 128 + pr];
          out[jj] = dim < half ? v[jj] * c - pv * s : v[jj] * c + pv * s;
        }
      }
      named_bar_sync(1, 128);
    } else {
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) out[jj] = v[jj];
    }
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
      const int j = j0 + jj;
      if (j >= e.M) continue;
      if (sec == 0) {
        p.q_out[static_cast<size_t>(j) * d + f] = __float2bfloat16_rn(out[jj]);
      } else {
        const int m = batch_row(e, j);
        const int b = st->row_req[m];
        const int crow = st->req_ctx[b] + (m - st->req_rowoff[b]);
        __nv_bfloat16* kv = st->kv_layer[e.layer];
        const size_t off =
            ((static_cast<size_t>(st->req_slot[b]) * 2 + (sec - 1)) * p.n_heads + head) * static_cast<size_t>(st->kv_cap) +
            crow;
        kv[off * D + dim] = __float2bfloat16_rn(out[jj]);
      }
    }
  } else if constexpr (EPI == kEpiSwiglu) {
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) e.xch[jj * 128 + r] = v[jj];
    named_bar_sync(1, 128);
    if (r < 64) {
      const int fcol = t * 64 + r;
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) {
        const int j = j0 + jj;
        if (j < e.M) {
          const float g = v[jj];
          const float u = e.xch[jj * 128 + r + 64];
          p.act_out[static_cast<size_t>(j) * p.act_ld + fcol] = __float2bfloat16_rn(g / (1.f + expf(-g)) * u);
        }
      }
    }
    named_bar_sync(1, 128);
  } else if constexpr (EPI == kEpiLmHead) {
    const int o = t * 128 + r;
    const bool valid = o < p.vocab;
    float* logits = p.step ? p.step->logits : nullptr;
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
      const int j = j0 + jj;
      float val = valid ? v[jj] : -INFINITY;
      if (valid && j < e.M) {
        if (logits) logits[static_cast<size_t>(batch_row(e, j)) * p.vocab + o] = v[jj];
        if (v[jj] != v[jj]) report(p.status, kStatusCheck);
      }
      int idx = o;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, val, off);
        const int oi = __shfl_xor_sync(0xffffffffu, idx, off);
        if (ov > val || (ov == val && oi < idx)) {
          val = ov;
          idx = oi;
        }
      }
      if (e.lane == 0) {
        e.redv[e.q * 16 + jj] = val;
        e.redi[e.q * 16 + jj] = idx;
      }
    }
    named_bar_sync(1, 128);
    if (e.et < 16) {
      const int jj = e.et, j = j0 + jj;
      float bv = e.redv[jj];
      int bi = e.redi[jj];
#pragma unroll
      for (int w = 1; w < 4; ++w) {
        const float ov = e.redv[w * 16 + jj];
        const int oi = e.redi[w * 16 + jj];
        if (ov > bv || (ov == bv && oi < bi)) {
          bv = ov;
          bi = oi;
        }
      }
      if (j < e.M) {
        p.amax_val[static_cast<size_t>(t) * kMaxRows + batch_row(e, j)] = bv;
        p.amax_idx[static_cast<size_t>(t) * kMaxRows + batch_row(e, j)] = bi;
      }
    }
    named_bar_sync(1, 128);
  }
}

template <int EPI>
__global__ void __launch_bounds__(kGemmThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX, const GemmParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int S = p.stages;
  const int n_pad = p.n_pad;
  const uint32_t x_bytes = static_cast<uint32_t>(n_pad) * 128u;
  uint8_t* sW = base;
  uint8_t* sX = base + static_cast<size_t>(S) * kWTileBytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sX + static_cast<size_t>(S) * x_bytes);
  uint64_t* empty = full + S;
  uint64_t* accf = empty + S;
  uint64_t* acce = accf + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acce + 2);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  int* bcast = reinterpret_cast<int*>(tmem_slot + 2);  // [3]
  float* xch = reinterpret_cast<float*>(tmem_slot + 16);
  float* redv = xch + 16 * 128;
  int* redi = reinterpret_cast<int*>(redv + 64);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t ncols = gemm_tmem_cols(n_pad, p.n_acc_bufs);

  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&accf[i], 1);
      mbar_init(&acce[i], 128);
    }
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tmW);
    prefetch_tmap(&tmX);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, ncols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const long long T = static_cast<long long>(p.n_tiles) * p.kb;
  const int G = gridDim.x, c = blockIdx.x;
  const long long it0 = T * c / G, it1 = T * (c + 1) / G;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer ----------------
      // The plan was written by the controller, several kernels upstream: every kernel triggers its
      // dependents only after its own griddepcontrol.wait, so that kernel has completed here.
      int layer = p.layer_fixed;
      if (layer < 0) layer = p.slot < p.plan->n_act ? p.plan->act_layer[p.slot] : 0;
      const long long n_it = it1 - it0;
      const int pre = static_cast<int>(n_it < S ? n_it : S);
      for (int i = 0; i < pre; ++i) {
        const long long it = it0 + i;
        const int t = static_cast<int>(it / p.kb), kk = static_cast<int>(it % p.kb);
        mbar_arrive_expect_tx(&full[i], kWTileBytes + x_bytes);
        if (p.w_tiled)
          bulk_load(sW + static_cast<size_t>(i) * kWTileBytes,
                    p.w_tiled + layer * p.w_layer_elems + (static_cast<size_t>(t) * p.kb + kk) * kTileElems, kWTileBytes,
                    &full[i]);
        else
          tma_load_3d(sW + static_cast<size_t>(i) * kWTileBytes, &tmW, &full[i], kk * 64, t * 128, layer);
      }
      griddep_wait();
      griddep_launch();
      for (int i = 0; i < pre; ++i) {
        const int kk = static_cast<int>((it0 + i) % p.kb);
        tma_load_2d(sX + static_cast<size_t>(i) * x_bytes, &tmX, &full[i], kk * 64, 0);
      }
      for (long long i = pre; i < n_it; ++i) {
        const int s = static_cast<int>(i % S);
        const uint32_t ph = static_cast<uint32_t>((i / S) & 1) ^ 1u;
        if (!mbar_wait(&empty[s], ph, abort_flag, p.status)) break;
        const long long it = it0 + i;
        const int t = static_cast<int>(it / p.kb), kk = static_cast<int>(it % p.kb);
        mbar_arrive_expect_tx(&full[s], kWTileBytes + x_bytes);
        if (p.w_tiled)
          bulk_load(sW + static_cast<size_t>(s) * kWTileBytes,
                    p.w_tiled + layer * p.w_layer_elems + (static_cast<size_t>(t) * p.kb + kk) * kTileElems, kWTileBytes,
                    &full[s]);
        else
          tma_load_3d(sW + static_cast<size_t>(s) * kWTileBytes, &tmW, &full[s], kk * 64, t * 128, layer);
        tma_load_2d(sX + static_cast<size_t>(s) * x_bytes, &tmX, &full[s], kk * 64, 0);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      griddep_wait();
      griddep_launch();
      const uint32_t idesc = idesc_bf16_m128(n_pad);
      long long it = it0, i = 0;
      int t, k0, k1, use = 0;
      bool ok = true;
      while (ok && next_segment(it, it1, p.kb, t, k0, k1)) {
        const int buf = p.n_acc_bufs == 2 ? (use & 1) : 0;
        const int ub = p.n_acc_bufs == 2 ? (use >> 1) : use;
        if (!mbar_wait(&acce[buf], static_cast<uint32_t>(ub & 1) ^ 1u, abort_flag, p.status)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(buf * n_pad);
        for (int kk = k0; kk < k1; ++kk, ++i) {
          const int s = static_cast<int>(i % S);
          if (!mbar_wait(&full[s], static_cast<uint32_t>((i / S) & 1), abort_flag, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t a0 = smem_u32(sW + static_cast<size_t>(s) * kWTileBytes);
          const uint32_t b0 = smem_u32(sX + static_cast<size_t>(s) * x_bytes);
#pragma unroll
          for (int k16 = 0; k16 < 4; ++k16) {
            umma_bf16(d_tmem, sdesc_sw128(a0 + k16 * 32), sdesc_sw128(b0 + k16 * 32), idesc,
                      (kk > k0 || k16 > 0) ? 1u : 0u);
          }
          umma_commit(&empty[s]);
        }
        if (!ok) break;
        umma_commit(&accf[buf]);
        ++use;
      }
    }
  } else {
    // ---------------- epilogue warps ----------------
    griddep_wait();
    griddep_launch();
    EpiCtx e;
    e.q = warp & 3;
    e.lane = lane;
    e.et = threadIdx.x - 64;
    e.xch = xch;
    e.redv = redv;
    e.redi = redi;
    if (p.slot >= 0) {
      // A slot beyond the controller's layer count (host/device disagreement, already reported
      // by the controller) writes nothing.
      const bool live = p.slot == kFinalSlot || p.slot < p.plan->n_act;
      e.M = live ? p.plan->slot_M[p.slot] : 0;
      e.rows = p.plan->slot_rows[p.slot];
      e.layer = (live && p.slot < kFinalSlot) ? p.plan->act_layer[p.slot] : -1;
    } else {
      e.M = p.m_raw;
      e.rows = nullptr;
      e.layer = p.layer_fixed;
    }
    const int r = e.q * 32 + lane;
    long long it = it0;
    int t, k0, k1, use = 0;
    while (next_segment(it, it1, p.kb, t, k0, k1)) {
      const int buf = p.n_acc_bufs == 2 ? (use & 1) : 0;
      const int ub = p.n_acc_bufs == 2 ? (use >> 1) : use;
      if (!mbar_wait(&accf[buf], static_cast<uint32_t>(ub & 1), abort_flag, p.status)) break;
      tc_fence_after();
      const uint32_t tb = tmem_base + (static_cast<uint32_t>(e.q * 32) << 16) + static_cast<uint32_t>(buf * n_pad);
      const int n_ch = n_pad >> 4;
      if (k0 == 0 && k1 == p.kb) {
        for (int ch = 0; ch < n_ch; ++ch) {
          float v[16];
          tmem_ld16(tb + ch * 16, v);
          epilogue_chunk<EPI>(p, e, t, r, ch, v);
        }
        tc_fence_before();
        mbar_arrive(&acce[buf]);
      } else {
        float* part = p.partials + static_cast<size_t>(c + t) * 128 * n_pad;
        for (int ch = 0; ch < n_ch; ++ch) {
          float v[16];
          tmem_ld16(tb + ch * 16, v);
#pragma unroll
          for (int jj = 0; jj < 16; ++jj) __stcg(&part[(ch * 16 + jj) * 128 + r], v[jj]);
        }
        tc_fence_before();
        mbar_arrive(&acce[buf]);
        named_bar_sync(1, 128);  // every thread's partial stores precede the release below
        if (e.et == 0) {
          const int cf = cta_of(static_cast<long long>(t) * p.kb, T, G);
          const int cl = cta_of(static_cast<long long>(t + 1) * p.kb - 1, T, G);
          const int old = atom_add_acq_rel_gpu(&p.counters[t], 1);
          const int last = old == cl - cf;
          if (last) atomicExch(&p.counters[t], 0);
          bcast[0] = last;
          bcast[1] = cf;
          bcast[2] = cl;
        }
        named_bar_sync(1, 128);
        if (bcast[0]) {  // (the counter's acquire, then the barrier: the other partials are visible)
          const int cf = bcast[1], cl = bcast[2];
          for (int ch = 0; ch < n_ch; ++ch) {
            float v[16];
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) v[jj] = 0.f;
            for (int cc = cf; cc <= cl; ++cc) {
              const float* pp = p.partials + static_cast<size_t>(cc + t) * 128 * n_pad;
#pragma unroll
              for (int jj = 0; jj < 16; ++jj) v[jj] += __ldcg(&pp[(ch * 16 + jj) * 128 + r]);
            }
            epilogue_chunk<EPI>(p, e, t, r, ch, v);
          }
        }
        named_bar_sync(1, 128);
      }
      ++use;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, ncols);
  }
}

template <int EPI>
cudaError_t gemm_max_carveout() {
  return cudaFuncSetAttribute(gemm_kernel<EPI>, cudaFuncAttributePreferredSharedMemoryCarveout,
                              cudaSharedmemCarveoutMaxShared);
}

cudaError_t gemm_prepare(size_t max_smem) {
  cudaError_t e;
  const int bytes = static_cast<int>(max_smem);
  // One shared-memory carveout for every kernel of the step: no L1/shared reconfiguration at
  // kernel boundaries.
  if ((e = gemm_max_carveout<kEpiStore>()) || (e = gemm_max_carveout<kEpiQkv>()) || (e = gemm_max_carveout<kEpiResid>()) ||
      (e = gemm_max_carveout<kEpiSwiglu>()) || (e = gemm_max_carveout<kEpiLmHead>()))
    return e;
  if ((e = cudaFuncSetAttribute(gemm_kernel<kEpiStore>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes))) return e;
  if ((e = cudaFuncSetAttribute(gemm_kernel<kEpiQkv>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes))) return e;
  if ((e = cudaFuncSetAttribute(gemm_kernel<kEpiResid>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes))) return e;
  if ((e = cudaFuncSetAttribute(gemm_kernel<kEpiSwiglu>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes))) return e;
  return cudaFuncSetAttribute(gemm_kernel<kEpiLmHead>, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

cudaError_t launch_gemm(int epi, const CUtensorMap& tmW, const CUtensorMap& tmX, const GemmParams& p, int grid,
                        size_t smem, cudaStream_t s, bool pdl) {
  const dim3 g(grid), b(kGemmThreads);
  switch (epi) {
    case kEpiStore: return launch_k(gemm_kernel<kEpiStore>, g, b, smem, s, pdl, tmW, tmX, p);
    case kEpiQkv: return launch_k(gemm_kernel<kEpiQkv>, g, b, smem, s, pdl, tmW, tmX, p);
    case kEpiResid: return launch_k(gemm_kernel<kEpiResid>, g, b, smem, s, pdl, tmW, tmX, p);
    case kEpiSwiglu: return launch_k(gemm_kernel<kEpiSwiglu>, g, b, smem, s, pdl, tmW, tmX, p);
    case kEpiLmHead: return launch_k(gemm_kernel<kEpiLmHead>, g, b, smem, s, pdl, tmW, tmX, p);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace tss
