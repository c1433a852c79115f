// Persistent verify kernel: every active layer of a verification step plus the LM head in one
// cooperative launch, one CTA per SM.
//
// The step is a fixed sequence of GEMM phases -- for each layer of the union (ascending):
// QKV, O, gate/up, down; then the LM head -- with the attention of a layer between its QKV and
// O phases.  Each phase is split stream-K over the grid exactly as in gemm.cu.  Per CTA:
//
//   warp 0      TMA producer of weight tiles.  It walks the whole phase sequence and never waits
//               for activations, so the weight stream does not stop at phase boundaries (it is
//               bounded only by the shared-memory ring).
//   warp 1      tcgen05.mma issuer (accumulators in TMEM, double-buffered).
//   warp 2      B-operand producer: for every k-block it waits until the activations it needs
//               are final, then writes the N x 64 bf16 tile (128-byte swizzle) -- from h times the
//               RMSNorm gain for QKV / gate-up / LM head, by TMA from the attention output or the
//               SwiGLU activations for O / down.
//   warps 4-7   epilogues (TMEM -> registers, stream-K fixup, fused op) and the attention items.
//
// Phases hand data over through global memory and per-tile flags stamped with a sequence
// number that grows monotonically over the step and across steps (seq = epoch*1024 + 8*(slot+1)
// + kind), so flags are never reset.  A consumer waits only for the producer tiles it reads:
// a k-block of QKV / gate-up / LM head needs one 128-feature tile of h; an O k-block needs the
// attention output of one head for every request; a down k-block needs one gate/up tile.
// The RMSNorm is split accordingly: the B operand is bf16(h * g), and the per-row factor
// 1/sqrt(mean(h^2) + eps) is applied to the accumulator in the epilogue, from per-tile partial
// sums of squares written by the residual epilogues.
//
// Every wait is bounded (2 s); on expiry the kernel records TIMEOUT, raises a grid-wide abort
// word and all roles leave their loops.
#include "attn_body.cuh"

namespace tss {

constexpr int kMkThreads = 256;
constexpr uint32_t kMkWBytes = 128 * 64 * 2;

enum MkKind : int { kMkQkv = 1, kMkAtt = 2, kMkO = 3, kMkGu = 4, kMkDown = 5, kMkLm = 6 };

__device__ __forceinline__ unsigned long long mk_seq(unsigned long long base, int slot, int kind) {
  return base + static_cast<unsigned long long>(slot + 1) * 8ull + static_cast<unsigned long long>(kind);
}

__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}
__device__ __forceinline__ void st_release_u64(unsigned long long* p, unsigned long long v) {
  asm volatile("st.release.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}
__device__ __forceinline__ void fence_proxy_async_shared() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Barrier over `n` threads that also returns the AND of every thread's `v` (uniform result).
__device__ __forceinline__ bool bar_and(int id, int n, bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 q, %3, 0;\n\t"
      "bar.red.and.pred p, %1, %2, q;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(r)
      : "r"(id), "r"(n), "r"(static_cast<uint32_t>(v))
      : "memory");
  return r != 0;
}

struct MkShared {
  volatile int* abort_s;
  int* abort_g;
  int* status;
};

__device__ __forceinline__ bool mk_aborted(const MkShared& sh) {
  if (*sh.abort_s) return true;
  if (*reinterpret_cast<volatile int*>(sh.abort_g)) {
    *sh.abort_s = 1;
    return true;
  }
  return false;
}

__device__ __forceinline__ void mk_fail(const MkShared& sh) {
  *sh.abort_s = 1;
  atomicExch(sh.abort_g, 1);
  report(sh.status, kStatusTimeout);
}

// Bounded wait for *f >= target.
__device__ bool mk_wait_flag(const unsigned long long* f, unsigned long long target, const MkShared& sh) {
  if (ld_acquire_u64(f) >= target) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (ld_acquire_u64(f) >= target) return true;
    if ((i & 63) == 0) {
      if (mk_aborted(sh)) return false;
      if (globaltimer_ns() - t0 > kWaitLimitNs) {
        mk_fail(sh);
        return false;
      }
    }
    __nanosleep(64);
  }
}

// Bounded mbarrier wait that also leaves when another CTA aborted.
__device__ bool mk_wait_bar(uint64_t* bar, uint32_t parity, const MkShared& sh) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 255) == 0) {
      if (mk_aborted(sh)) return false;
      if (globaltimer_ns() - t0 > kWaitLimitNs) {
        mk_fail(sh);
        return false;
      }
    }
  }
}

struct MkPhase {
  int kind, slot, layer, n_tiles, kb;
};

__device__ __forceinline__ MkPhase mk_phase(const MkParams& p, const PlanDev* pl, int pi) {
  MkPhase ph;
  if (pi < 4 * p.n_act) {
    ph.slot = pi >> 2;
    ph.layer = pl->act_layer[ph.slot];
    switch (pi & 3) {
      case 0: ph.kind = kMkQkv; ph.n_tiles = 3 * p.d / 128; ph.kb = p.d / 64; break;
      case 1: ph.kind = kMkO; ph.n_tiles = p.d / 128; ph.kb = p.d / 64; break;
      case 2: ph.kind = kMkGu; ph.n_tiles = p.Ft; ph.kb = p.d / 64; break;
      default: ph.kind = kMkDown; ph.n_tiles = p.d / 128; ph.kb = p.F_pad / 64; break;
    }
  } else {
    ph.kind = kMkLm;
    ph.slot = p.n_act;
    ph.layer = 0;
    ph.n_tiles = p.V_pad / 128;
    ph.kb = p.d / 64;
  }
  return ph;
}

// CTA c's stream-K range of a phase over geff = min(grid, iterations) CTAs.
__device__ __forceinline__ void mk_range(const MkPhase& ph, int c, int G, long long& it0, long long& it1, int& geff) {
  const long long T = static_cast<long long>(ph.n_tiles) * ph.kb;
  geff = static_cast<int>(T < G ? T : G);
  if (c >= geff) {
    it0 = it1 = 0;
    return;
  }
  it0 = T * c / geff;
  it1 = T * (c + 1) / geff;
}

__device__ __forceinline__ int mk_cta_of(long long i, long long T, int G) {
  return static_cast<int>(((i + 1) * G - 1) / T);
}

__device__ __forceinline__ bool mk_next_segment(long long& it, long long end, int kb, int& t, int& k0, int& k1) {
  if (it >= end) return false;
  t = static_cast<int>(it / kb);
  k0 = static_cast<int>(it - static_cast<long long>(t) * kb);
  const long long tile_end = static_cast<long long>(t + 1) * kb;
  const long long e = end < tile_end ? end : tile_end;
  k1 = static_cast<int>(e - static_cast<long long>(t) * kb);
  it = e;
  return true;
}

// Slot whose compacted rows feed a phase (the LM head runs on all rows).
__device__ __forceinline__ int mk_row_slot(const MkPhase& ph) { return ph.kind == kMkLm ? kFinalSlot : ph.slot; }

// Sequence number h must have reached before a norm phase reads it (0: the embedding, i.e. the
// previous kernel, which has completed when this kernel starts).
__device__ __forceinline__ unsigned long long mk_h_dep(const MkParams& p, const MkPhase& ph) {
  if (ph.kind == kMkQkv) return ph.slot == 0 ? 0ull : mk_seq(p.seq_base, ph.slot - 1, kMkDown);
  if (ph.kind == kMkGu) return mk_seq(p.seq_base, ph.slot, kMkO);
  return p.n_act == 0 ? 0ull : mk_seq(p.seq_base, p.n_act - 1, kMkDown);  // LM head
}

struct MkEpi {
  int M;
  const int* rows;
  float* xch;    // [16][128]
  float* redv;   // [4][16]
  int* redi;     // [4][16]
  float* rs;     // [kMaxRows] per-row RMSNorm factors of the current tile
  int q, lane, et;
};

// Wait until every 128-feature tile of h has reached `dep`, then compute the RMSNorm factors of
// the phase's rows from the partial sums of squares (fixed order, deterministic).
__device__ bool mk_prepare_rs(const MkParams& p, const MkEpi& e, unsigned long long dep, const MkShared& sh) {
  const int nt = p.d / 128;
  bool ok = true;
  for (int t = e.et; dep != 0ull && t < nt && ok; t += 128) ok = mk_wait_flag(&p.hflag[t], dep, sh);
  if (!bar_and(1, 128, ok)) return false;
  for (int j = e.et; j < e.M; j += 128) {
    const int m = e.rows[j];
    float ss = 0.f;
    for (int t = 0; t < nt; ++t) ss += __ldcg(&p.ssp[static_cast<size_t>(t) * kMaxRows + m]);
    e.rs[j] = rsqrtf(ss / static_cast<float>(p.d) + p.eps);
  }
  named_bar_sync(1, 128);
  return true;
}

// Fused epilogue of one 16-token chunk (tokens ch*16 ..) of output row r of tile t.
__device__ void mk_epilogue_chunk(const MkParams& p, const MkPhase& ph, const MkEpi& e, int t, int r, int ch,
                                  const float* v) {
  const StepDesc* st = p.step;
  const int j0 = ch * 16;
  if (ph.kind == kMkQkv) {
    const int d = p.d, D = p.D, half = D >> 1;
    const int o = t * 128 + r;
    const int sec = o / d;
    const int f = o - sec * d;
    const int head = f / D, dim = f - head * D;
    float val[16];
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) val[jj] = j0 + jj < e.M ? v[jj] * e.rs[j0 + jj] : 0.f;
    if (sec < 2) {
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) e.xch[jj * 128 + r] = val[jj];
      named_bar_sync(1, 128);
      const int pr = r ^ half;
      const int i = dim & (half - 1);
      float rot[16];
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) {
        rot[jj] = 0.f;
        if (j0 + jj < e.M) {
          const int pos = st->row_pos[e.rows[j0 + jj]];
          const float c = p.rope_cos[static_cast<size_t>(pos) * half + i];
          const float s = p.rope_sin[static_cast<size_t>(pos) * half + i];
          const float pv = e.xch[jj * 128 + pr];
          rot[jj] = dim < half ? val[jj] * c - pv * s : val[jj] * c + pv * s;
        }
      }
      named_bar_sync(1, 128);
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) val[jj] = rot[jj];
    }
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
      const int j = j0 + jj;
      if (j >= e.M) continue;
      if (sec == 0) {
        p.qbuf[static_cast<size_t>(j) * d + f] = __float2bfloat16_rn(val[jj]);
      } else {
        const int m = e.rows[j];
        const int b = st->row_req[m];
        const int crow = st->req_ctx[b] + (m - st->req_rowoff[b]);
        const size_t off =
            ((static_cast<size_t>(st->req_slot[b]) * 2 + (sec - 1)) * p.H + head) * static_cast<size_t>(st->kv_cap) + crow;
        st->kv_layer[ph.layer][off * D + dim] = __float2bfloat16_rn(val[jj]);
      }
    }
  } else if (ph.kind == kMkO || ph.kind == kMkDown) {
    // residual add, then this tile's partial sum of squares of the updated rows
    const int o = t * 128 + r;
    float sq[16];
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
      const int j = j0 + jj;
      sq[jj] = 0.f;
      if (j < e.M) {
        float* hp = p.h + static_cast<size_t>(e.rows[j]) * p.d + o;
        const float nv = __ldcg(hp) + v[jj];
        *hp = nv;
        sq[jj] = nv * nv;
      }
    }
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) sq[jj] += __shfl_xor_sync(0xffffffffu, sq[jj], off);
    }
    if (e.lane == 0) {
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) e.redv[e.q * 16 + jj] = sq[jj];
    }
    named_bar_sync(1, 128);
    if (e.et < 16 && j0 + e.et < e.M) {
      const int jj = e.et;
      const float s4 = (e.redv[jj] + e.redv[16 + jj]) + (e.redv[32 + jj] + e.redv[48 + jj]);
      p.ssp[static_cast<size_t>(t) * kMaxRows + e.rows[j0 + jj]] = s4;
    }
    named_bar_sync(1, 128);
  } else if (ph.kind == kMkGu) {
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) e.xch[jj * 128 + r] = v[jj];
    named_bar_sync(1, 128);
    if (r < 64) {
      const int fcol = t * 64 + r;
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) {
        const int j = j0 + jj;
        if (j < e.M) {
          const float g = v[jj] * e.rs[j];
          const float u = e.xch[jj * 128 + r + 64] * e.rs[j];
          p.act[static_cast<size_t>(j) * p.F_pad + fcol] = __float2bfloat16_rn(g / (1.f + expf(-g)) * u);
        }
      }
    }
    named_bar_sync(1, 128);
  } else {  // LM head: logits (optional) and per-tile argmax, lowest index on ties
    const int o = t * 128 + r;
    const bool valid = o < p.V;
    float* logits = st->logits;
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
      const int j = j0 + jj;
      float val = -INFINITY;
      if (valid && j < e.M) {
        val = v[jj] * e.rs[j];
        if (logits) logits[static_cast<size_t>(e.rows[j]) * p.V + o] = val;
        if (val != val) report(p.status, kStatusCheck);
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
    if (e.et < 16 && j0 + e.et < e.M) {
      const int jj = e.et;
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
      p.amax_val[static_cast<size_t>(t) * kMaxRows + e.rows[j0 + jj]] = bv;
      p.amax_idx[static_cast<size_t>(t) * kMaxRows + e.rows[j0 + jj]] = bi;
    }
    named_bar_sync(1, 128);
  }
}

__device__ __forceinline__ unsigned long long* mk_tile_flag(const MkParams& p, int kind, int t) {
  switch (kind) {
    case kMkQkv: return p.qkvflag + t;
    case kMkGu: return p.guflag + t;
    case kMkO:
    case kMkDown: return p.hflag + t;
    default: return nullptr;
  }
}

template <int D>
__global__ void __launch_bounds__(kMkThreads, 1)
    verify_mk_kernel(const __grid_constant__ CUtensorMap tm_qkv, const __grid_constant__ CUtensorMap tm_o,
                     const __grid_constant__ CUtensorMap tm_gu, const __grid_constant__ CUtensorMap tm_down,
                     const __grid_constant__ CUtensorMap tm_lm, const __grid_constant__ CUtensorMap tm_xo,
                     const __grid_constant__ CUtensorMap tm_xact, const MkParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int S = p.stages, n_pad = p.n_pad;
  const uint32_t x_bytes = static_cast<uint32_t>(n_pad) * 128u;
  uint8_t* sW = base;
  uint8_t* sX = sW + static_cast<size_t>(S) * kMkWBytes;
  uint8_t* s_attn = sX + static_cast<size_t>(S) * x_bytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(s_attn + attn_smem_bytes_impl(D));
  uint64_t* empty = full + S;
  uint64_t* accf = empty + S;
  uint64_t* acce = accf + 2;
  int* misc = reinterpret_cast<int*>(acce + 2);  // [0] tmem addr, [1] abort, [2..4] bcast, [5] s_last
  float* xch = reinterpret_cast<float*>(misc + 16);
  float* redv = xch + 16 * 128;
  int* redi = reinterpret_cast<int*>(redv + 64);
  float* rs = reinterpret_cast<float*>(redi + 64);
  float (*sM)[16] = reinterpret_cast<float (*)[16]>(rs + kMaxRows);
  float (*sL)[16] = reinterpret_cast<float (*)[16]>(rs + kMaxRows + 64);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t ncols = gemm_tmem_cols(n_pad, 2);
  const PlanDev* pl = p.plan;
  MkShared sh;
  sh.abort_s = reinterpret_cast<volatile int*>(misc + 1);
  sh.abort_g = p.abort_word;
  sh.status = p.status;

  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(&full[i], 2);  // weight TMA arrival + B-operand arrival
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&accf[i], 1);
      mbar_init(&acce[i], 128);
    }
    *sh.abort_s = 0;
    fence_mbar_init();
    prefetch_tmap(&tm_qkv);
    prefetch_tmap(&tm_o);
    prefetch_tmap(&tm_gu);
    prefetch_tmap(&tm_down);
    prefetch_tmap(&tm_lm);
    prefetch_tmap(&tm_xo);
    prefetch_tmap(&tm_xact);
  }
  if (warp == 1) {
    tmem_alloc(reinterpret_cast<uint32_t*>(misc), ncols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = static_cast<uint32_t>(misc[0]);
  griddep_wait();  // the controller's plan and the embedding are complete

  const int G = gridDim.x, c = blockIdx.x;
  // A host/device disagreement on the layer union (reported by the controller) runs nothing.
  const int n_phases = pl->n_act == p.n_act ? 4 * p.n_act + 1 : 0;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- weight TMA producer: never waits for activations ----------------
      long long i = 0;
      bool ok = true;
      for (int pi = 0; ok && pi < n_phases; ++pi) {
        const MkPhase ph = mk_phase(p, pl, pi);
        long long it0, it1;
        int geff;
        mk_range(ph, c, G, it0, it1, geff);
        const CUtensorMap* tm = ph.kind == kMkQkv ? &tm_qkv
                                : ph.kind == kMkO ? &tm_o
                                : ph.kind == kMkGu ? &tm_gu
                                : ph.kind == kMkDown ? &tm_down
                                                     : &tm_lm;
        for (long long it = it0; it < it1; ++it, ++i) {
          const int s = static_cast<int>(i % S);
          if (!mk_wait_bar(&empty[s], static_cast<uint32_t>((i / S) & 1) ^ 1u, sh)) {
            ok = false;
            break;
          }
          const int t = static_cast<int>(it / ph.kb), kk = static_cast<int>(it % ph.kb);
          mbar_arrive_expect_tx(&full[s], kMkWBytes);
          tma_load_3d(sW + static_cast<size_t>(s) * kMkWBytes, tm, &full[s], kk * 64, t * 128, ph.layer);
        }
      }
      if (!ok) {  // let weight tiles already in flight land before the CTA can exit
        const uint64_t t0 = globaltimer_ns();
        while (globaltimer_ns() - t0 < 50000) {
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer ----------------
      const uint32_t idesc = idesc_bf16_m128(n_pad);
      long long i = 0;
      int use = 0;
      bool ok = true;
      for (int pi = 0; ok && pi < n_phases; ++pi) {
        const MkPhase ph = mk_phase(p, pl, pi);
        long long it0, it1;
        int geff;
        mk_range(ph, c, G, it0, it1, geff);
        long long it = it0;
        int t, k0, k1;
        while (ok && mk_next_segment(it, it1, ph.kb, t, k0, k1)) {
          const int buf = use & 1;
          if (!mk_wait_bar(&acce[buf], static_cast<uint32_t>((use >> 1) & 1) ^ 1u, sh)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(buf * n_pad);
          for (int kk = k0; kk < k1; ++kk, ++i) {
            const int s = static_cast<int>(i % S);
            if (!mk_wait_bar(&full[s], static_cast<uint32_t>((i / S) & 1), sh)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t a0 = smem_u32(sW + static_cast<size_t>(s) * kMkWBytes);
            const uint32_t b0 = smem_u32(sX + static_cast<size_t>(s) * x_bytes);
#pragma unroll
            for (int k16 = 0; k16 < 4; ++k16)
              umma_bf16(d_tmem, sdesc_sw128(a0 + k16 * 32), sdesc_sw128(b0 + k16 * 32), idesc,
                        (kk > k0 || k16 > 0) ? 1u : 0u);
            umma_commit(&empty[s]);
          }
          if (!ok) break;
          umma_commit(&accf[buf]);
          ++use;
        }
      }
    }
  } else if (warp == 2) {
    // ---------------- B-operand producer ----------------
    long long i = 0;
    bool ok = true;
    for (int pi = 0; ok && pi < n_phases; ++pi) {
      const MkPhase ph = mk_phase(p, pl, pi);
      long long it0, it1;
      int geff;
      mk_range(ph, c, G, it0, it1, geff);
      if (it0 >= it1) continue;
      const int rslot = mk_row_slot(ph);
      const int M = pl->slot_M[rslot];
      const int* rows = pl->slot_rows[rslot];
      const unsigned long long hdep = (ph.kind == kMkO || ph.kind == kMkDown) ? 0ull : mk_h_dep(p, ph);
      const float* gain = ph.kind == kMkQkv  ? p.g_attn + static_cast<size_t>(ph.layer) * p.d
                          : ph.kind == kMkGu ? p.g_mlp + static_cast<size_t>(ph.layer) * p.d
                                             : p.g_final;
      int ready_dep = -1;  // last dependency index already seen complete
      for (long long it = it0; ok && it < it1; ++it, ++i) {
        const int s = static_cast<int>(i % S);
        const int kk = static_cast<int>(it % ph.kb);
        if (lane == 0) ok = mk_wait_bar(&empty[s], static_cast<uint32_t>((i / S) & 1) ^ 1u, sh);
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) break;
        // dependency of this k-block
        if (ph.kind == kMkO) {
          const int head = kk * 64 / p.D;
          if (head != ready_dep) {
            const unsigned long long want = mk_seq(p.seq_base, ph.slot, kMkAtt);
            bool good = true;
            for (int b = lane; b < p.B; b += 32)
              if (pl->slot_crow[ph.slot][b] >= 0) good = good && mk_wait_flag(&p.attflag[b * p.H + head], want, sh);
            ok = __all_sync(0xffffffffu, good);
            ready_dep = head;
          }
        } else if (ph.kind == kMkDown) {
          if (kk != ready_dep) {
            if (lane == 0) ok = mk_wait_flag(&p.guflag[kk], mk_seq(p.seq_base, ph.slot, kMkGu), sh);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            ready_dep = kk;
          }
        } else if (hdep != 0ull) {
          const int ht = kk >> 1;  // 128-feature tile of h holding this k-block
          if (ht != ready_dep) {
            if (lane == 0) ok = mk_wait_flag(&p.hflag[ht], hdep, sh);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            ready_dep = ht;
          }
        }
        if (!ok) break;
        if (ph.kind == kMkO || ph.kind == kMkDown) {
          if (lane == 0) {
            fence_proxy_async_global();
            mbar_arrive_expect_tx(&full[s], x_bytes);
            tma_load_2d(sX + static_cast<size_t>(s) * x_bytes, ph.kind == kMkO ? &tm_xo : &tm_xact, &full[s], kk * 64, 0);
          }
        } else {
          uint8_t* xs = sX + static_cast<size_t>(s) * x_bytes;
          for (int idx = lane; idx < n_pad * 8; idx += 32) {
            const int row = idx >> 3, c8 = idx & 7;
            uint4 out = make_uint4(0, 0, 0, 0);
            if (row < M) {
              const float* hp = p.h + static_cast<size_t>(rows[row]) * p.d + kk * 64 + c8 * 8;
              const float* gp = gain + kk * 64 + c8 * 8;
              const float4 a = __ldcg(reinterpret_cast<const float4*>(hp));
              const float4 b = __ldcg(reinterpret_cast<const float4*>(hp + 4));
              const float4 ga = *reinterpret_cast<const float4*>(gp);
              const float4 gb = *reinterpret_cast<const float4*>(gp + 4);
              out.x = pack_bf16(a.x * ga.x, a.y * ga.y);
              out.y = pack_bf16(a.z * ga.z, a.w * ga.w);
              out.z = pack_bf16(b.x * gb.x, b.y * gb.y);
              out.w = pack_bf16(b.z * gb.z, b.w * gb.w);
            }
            *reinterpret_cast<uint4*>(xs + row * 128 + ((c8 ^ (row & 7)) << 4)) = out;
          }
          fence_proxy_async_shared();
          __syncwarp();
          if (lane == 0) mbar_arrive(&full[s]);
        }
      }
    }
  } else if (warp >= 4) {
    // ---------------- epilogues and attention ----------------
    MkEpi e;
    e.q = warp & 3;
    e.lane = lane;
    e.et = threadIdx.x - 128;
    e.xch = xch;
    e.redv = redv;
    e.redi = redi;
    e.rs = rs;
    const int r = e.q * 32 + lane;
    int* bcast = misc + 2;
    int use = 0;
    bool ok = true;
    AttnParams ap{};
    ap.n_splits = p.attn_splits;
    ap.n_heads = p.H;
    ap.d_model = p.d;
    ap.head_dim = D;
    ap.scale_log2 = p.scale_log2;
    ap.plan = pl;
    ap.step = p.step;
    ap.q = p.qbuf;
    ap.o = p.obuf;
    ap.part_o = p.attn_po;
    ap.part_ml = p.attn_pml;
    ap.counters = p.attn_cnt;
    ap.status = p.status;
    for (int pi = 0; ok && pi < n_phases; ++pi) {
      const MkPhase ph = mk_phase(p, pl, pi);
      long long it0, it1;
      int geff;
      mk_range(ph, c, G, it0, it1, geff);
      const int rslot = mk_row_slot(ph);
      e.M = pl->slot_M[rslot];
      e.rows = pl->slot_rows[rslot];
      const long long T = static_cast<long long>(ph.n_tiles) * ph.kb;
      float* partials = (pi & 1) ? p.partials1 : p.partials0;
      int* counters = p.counters + static_cast<size_t>(ph.kind) * p.max_tiles;
      const bool needs_rs = ph.kind == kMkQkv || ph.kind == kMkGu || ph.kind == kMkLm;
      const unsigned long long hdep = needs_rs ? mk_h_dep(p, ph) : 0ull;
      long long it = it0;
      int t, k0, k1;
      while (ok && mk_next_segment(it, it1, ph.kb, t, k0, k1)) {
        const int buf = use & 1;
        const bool got = e.et == 0 ? mk_wait_bar(&accf[buf], static_cast<uint32_t>((use >> 1) & 1), sh) : true;
        if (!bar_and(1, 128, got)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t tb = tmem_base + (static_cast<uint32_t>(e.q * 32) << 16) + static_cast<uint32_t>(buf * n_pad);
        const int n_ch = n_pad >> 4;
        bool finalize = false;
        int cf = 0, cl = 0;
        if (k0 == 0 && k1 == ph.kb) {
          if (needs_rs && !mk_prepare_rs(p, e, hdep, sh)) {
            ok = false;
            break;
          }
          for (int ch = 0; ch < n_ch; ++ch) {
            float v[16];
            tmem_ld16(tb + ch * 16, v);
            mk_epilogue_chunk(p, ph, e, t, r, ch, v);
          }
          tc_fence_before();
          mbar_arrive(&acce[buf]);
          finalize = true;
        } else {
          float* part = partials + static_cast<size_t>(c + t) * 128 * n_pad;
          for (int ch = 0; ch < n_ch; ++ch) {
            float v[16];
            tmem_ld16(tb + ch * 16, v);
#pragma unroll
            for (int jj = 0; jj < 16; ++jj) __stcg(&part[(ch * 16 + jj) * 128 + r], v[jj]);
          }
          tc_fence_before();
          mbar_arrive(&acce[buf]);
          __threadfence();
          named_bar_sync(1, 128);
          if (e.et == 0) {
            const int f = mk_cta_of(static_cast<long long>(t) * ph.kb, T, geff);
            const int l = mk_cta_of(static_cast<long long>(t + 1) * ph.kb - 1, T, geff);
            const int old = atomicAdd(&counters[t], 1);
            const int last = old == l - f;
            if (last) atomicExch(&counters[t], 0);
            bcast[0] = last;
            bcast[1] = f;
            bcast[2] = l;
          }
          named_bar_sync(1, 128);
          finalize = bcast[0] != 0;
          cf = bcast[1];
          cl = bcast[2];
          named_bar_sync(1, 128);
          if (finalize) {
            __threadfence();
            if (needs_rs && !mk_prepare_rs(p, e, hdep, sh)) {
              ok = false;
              break;
            }
            for (int ch = 0; ch < n_ch; ++ch) {
              float v[16];
#pragma unroll
              for (int jj = 0; jj < 16; ++jj) v[jj] = 0.f;
              for (int cc = cf; cc <= cl; ++cc) {
                const float* pp = partials + static_cast<size_t>(cc + t) * 128 * n_pad;
#pragma unroll
                for (int jj = 0; jj < 16; ++jj) v[jj] += __ldcg(&pp[(ch * 16 + jj) * 128 + r]);
              }
              mk_epilogue_chunk(p, ph, e, t, r, ch, v);
            }
          }
        }
        if (finalize) {
          unsigned long long* flag = mk_tile_flag(p, ph.kind, t);
          __threadfence();
          named_bar_sync(1, 128);
          if (flag && e.et == 0) st_release_u64(flag, mk_seq(p.seq_base, ph.slot, ph.kind));
        }
        ++use;
      }
      if (!ok) break;
      if (ph.kind == kMkQkv) {
        // attention items of this layer: (request, head, split) round-robin over the grid
        ap.slot = ph.slot;
        const int per_req = p.H * p.attn_splits;
        const int n_items = p.B * per_req;
        const unsigned long long want = mk_seq(p.seq_base, ph.slot, kMkQkv);
        for (int item = c; ok && item < n_items; item += G) {
          const int b = item / per_req;
          const int head = (item - b * per_req) / p.attn_splits;
          const int split = item - b * per_req - head * p.attn_splits;
          if (pl->slot_crow[ph.slot][b] < 0) continue;
          bool good = true;
          if (e.et < 3) {
            const int tile = (e.et * p.d + head * D) / 128;
            good = mk_wait_flag(&p.qkvflag[tile], want, sh);
          }
          if (!bar_and(1, 128, good)) {
            ok = false;
            break;
          }
          const bool wrote = attention_item<D, 1>(ap, split, head, b, e.et, s_attn, sM, sL, misc + 5);
          if (wrote) {
            __threadfence();
            named_bar_sync(1, 128);
            if (e.et == 0) st_release_u64(&p.attflag[b * p.H + head], mk_seq(p.seq_base, ph.slot, kMkAtt));
          }
          named_bar_sync(1, 128);
        }
      }
    }
  }

  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, ncols);
  }
}

size_t mk_smem_bytes(int n_pad, int stages, int head_dim) {
  return 1024 + static_cast<size_t>(stages) * (kMkWBytes + static_cast<size_t>(n_pad) * 128) +
         attn_smem_bytes_impl(head_dim) + static_cast<size_t>(2 * stages + 4) * 8 + 64 + 16 * 128 * 4 + 64 * 4 * 2 +
         kMaxRows * 4 + 128 * 4 + 64;
}

cudaError_t mk_prepare() {
  cudaError_t e = cudaFuncSetAttribute(verify_mk_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, 232448);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(verify_mk_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, 232448);
  return e;
}

cudaError_t launch_verify_mk(const MkTensorMaps& tm, const MkParams& p, int grid, size_t smem, cudaStream_t s) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kMkThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;  // all CTAs co-resident: the dataflow waits need it
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (p.D == 64)
    return cudaLaunchKernelEx(&cfg, verify_mk_kernel<64>, tm.qkv, tm.o, tm.gu, tm.down, tm.lm, tm.xo, tm.xact, p);
  if (p.D == 128)
    return cudaLaunchKernelEx(&cfg, verify_mk_kernel<128>, tm.qkv, tm.o, tm.gu, tm.down, tm.lm, tm.xo, tm.xact, p);
  return cudaErrorInvalidValue;
}

int mk_max_blocks_per_sm(int head_dim, size_t smem) {
  int n = 0;
  if (head_dim == 64)
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, verify_mk_kernel<64>, kMkThreads, smem);
  else
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, verify_mk_kernel<128>, kMkThreads, smem);
  return n;
}

}  // namespace tss
