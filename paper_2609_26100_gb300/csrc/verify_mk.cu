// Persistent verify kernel: every active layer of a verification step plus the LM head in one
// cooperative launch, one CTA per SM.
//
// The step is a fixed sequence of GEMM phases -- for each layer of the union (ascending):
// QKV, O, gate/up, down; then the LM head -- with the attention of a layer between its QKV and
// O phases.  Each phase is split stream-K over the grid exactly as in gemm.cu.  Per CTA:
//
//   warp 0      TMA producer of weight tiles (lane 0).  It walks the whole phase sequence and
//               never waits for activations, so the weight stream does not stop at phase
//               boundaries (it is bounded only by the shared-memory ring).
//   warp 1      tcgen05.mma issuer (lane 0; accumulators in TMEM, up to 8 buffers).
//   warp 2      B-operand producer: for every k-block it waits until the activations it needs
//               are final (flags polled 32 at a time), then loads the N x 64 bf16 tile by TMA --
//               bf16(h * g) for QKV / gate-up / LM head, the attention output for O, the SwiGLU
//               activations for down.
//   warp 3      attention only.
//   warps 4-7   epilogues (TMEM -> registers, stream-K fixup, fused op).
// All roles run one loop over the phases; at each O phase (when the attention runs in this
// kernel) the eight warps first run the layer's attention items together, in the ring that every
// role has stopped using by then.
//
// Phases hand data over through global memory and per-tile flags stamped with a sequence
// number that grows monotonically over the step and across steps (seq = epoch*1024 + 8*(slot+1)
// + kind), so flags are never reset.  A consumer waits only for the producer tiles it reads:
// a k-block of QKV / gate-up / LM head needs one 128-feature tile of h; an O k-block needs the
// attention output of one head for every request; a down k-block needs one gate/up tile.
// The RMSNorm is split accordingly: the B operand is bf16(h * g) -- written, for the next norm
// phase, by the epilogue that finalises each 128-feature tile of h -- and the per-row factor
// 1/sqrt(mean(h^2) + eps) is applied to the accumulator in the epilogue, from per-tile partial
// sums of squares written by the same residual epilogues.
//
// Every wait is bounded (2 s by default, TSS_WAIT_LIMIT_MS at context creation); on expiry the
// kernel records TIMEOUT, raises a grid-wide abort word and all roles leave their loops.
#include "attn_body.cuh"

namespace tss {

constexpr int kMkThreads = 256;
constexpr int kMkMaxAcc = 8;  // TMEM accumulator buffers (fewer when N is large)

// Accumulator buffers for an MMA width: a power of two, at most 8, within 512 TMEM columns.
__host__ __device__ inline int mk_acc_bufs(int n_pad) {
  int nb = kMkMaxAcc;
  while (nb > 1 && nb * n_pad > 512) nb >>= 1;
  return nb;
}
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
  uint64_t limit_ns;  // bound of every wait (create-time setting, 2 s by default)
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
      if (globaltimer_ns() - t0 > sh.limit_ns) {
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
    if (mbar_try_wait_sleep(bar, parity, 20000u)) return true;
    if ((i & 255) == 0) {
      if (mk_aborted(sh)) return false;
      if (globaltimer_ns() - t0 > sh.limit_ns) {
        mk_fail(sh);
        return false;
      }
    }
  }
}

// Every thread of the CTA arrives on `bar` and waits (bounded) for all to arrive; n counts this
// thread's syncs on it (phase parity).
__device__ __forceinline__ bool mk_team_sync(uint64_t* bar, uint32_t& n, const MkShared& sh) {
  mbar_arrive(bar);
  const bool ok = mk_wait_bar(bar, n & 1u, sh);
  ++n;
  return ok;
}

struct MkPhase {
  int kind, slot, layer, n_tiles, kb;
};

// Optional timeline (TSS_TRACE): per CTA, per phase, the first and last activity of each role.
// trace[cta][pi * 8 + 2 * role + {0: first, 1: last}], roles 0 weight TMA, 1 B operand, 2 MMA,
// 3 epilogue; the attention of slot j at [kMkTracePhases * 8 + 2j + {0,1}].
constexpr int kMkTracePhases = 4 * kMaxLayers + 1;
constexpr int kMkTraceSub = kMkTracePhases * 8 + 2 * kMaxLayers;  // epilogue sub-steps of a phase's last segment
constexpr int kMkTraceAttn = kMkTraceSub + kMkTracePhases * 8;  // sub-steps of the slot-1 attention item
constexpr int kMkTraceSlots = kMkTraceAttn + 16;
__device__ __forceinline__ void mk_trace(const MkParams& p, int idx) {
  if (p.trace) p.trace[static_cast<size_t>(blockIdx.x) * kMkTraceSlots + idx] = globaltimer_ns();
}

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

// Pre-tiled weights of a phase's layer (blocks [tile][k-block] of 16 KiB).
__device__ __forceinline__ const __nv_bfloat16* mk_weights(const MkParams& p, const MkPhase& ph) {
  const size_t blocks = static_cast<size_t>(ph.n_tiles) * ph.kb;
  const __nv_bfloat16* base = ph.kind == kMkQkv ? p.w_qkv
                              : ph.kind == kMkO ? p.w_o
                              : ph.kind == kMkGu ? p.w_gu
                              : ph.kind == kMkDown ? p.w_down
                                                   : p.w_lm;
  return base + static_cast<size_t>(ph.layer) * blocks * kTileElems;
}

// CTA c's share of a phase as a sequence of segments (tile t, k-blocks [k0, k1)): stream-K over
// every iteration (tile x k-block) of the phase; or, when the phase has at least one tile per CTA
// and p.dp_tail is set, stream-K over its first n_tiles - G tiles followed by one whole tile per
// CTA, so that the phase ends with whole-tile epilogues (no partial tiles, no arrival counter,
// no reload of other CTAs' partials on its critical tail).  Residual phases keep plain stream-K.
struct MkSeg {
  long long it, it1;  // stream-K iterations of this CTA still to take
  long long T;        // stream-K iterations of the phase (the fix-up contributor arithmetic)
  int geff;           // CTAs sharing them
  int kb, whole;      // this CTA's whole tile after them, -1: none
  __device__ __forceinline__ bool next(int& t, int& k0, int& k1);
  __device__ __forceinline__ bool done() const { return it >= it1 && whole < 0; }
  __device__ __forceinline__ long long start() const { return it; }
};

__device__ __forceinline__ MkSeg mk_seg(const MkParams& p, const MkPhase& ph, int c, int G) {
  MkSeg s;
  s.kb = ph.kb;
  s.whole = -1;
  int n_split = ph.n_tiles;
  if (p.dp_tail && ph.n_tiles >= G && ph.kind != kMkO && ph.kind != kMkDown) {
    n_split = ph.n_tiles - G;
    s.whole = n_split + c;
  }
  s.T = static_cast<long long>(n_split) * ph.kb;
  s.geff = static_cast<int>(s.T < G ? s.T : G);
  if (c >= s.geff) {
    s.it = s.it1 = 0;
  } else {
    s.it = s.T * c / s.geff;
    s.it1 = s.T * (c + 1) / s.geff;
  }
  return s;
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

__device__ __forceinline__ bool MkSeg::next(int& t, int& k0, int& k1) {
  if (mk_next_segment(it, it1, kb, t, k0, k1)) return true;
  if (whole < 0) return false;
  t = whole;
  k0 = 0;
  k1 = kb;
  whole = -1;
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

// Accumulator values of tokens [16 ch, 16 ch + 16) of this thread's output row: W.hi + W.lo
// (the two parts are separate columns of one MMA when xs.parts == 1, already summed otherwise).
__device__ __forceinline__ void mk_acc_tokens(uint32_t tb, int ch, const XsLayout& xs, float* v) {
  if (xs.parts == 2) {
    tmem_ld16(tb + ch * 16, v);
  } else if (xs.half == 8) {  // up to 8 tokens: hi in columns 0..7, lo in 8..15
    float r[16];
    tmem_ld16(tb, r);
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) {
      v[jj] = r[jj] + r[8 + jj];
      v[8 + jj] = 0.f;
    }
  } else {
    float lo[16];
    tmem_ld16(tb + ch * 16, v);
    tmem_ld16(tb + xs.half + ch * 16, lo);
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) v[jj] += lo[jj];
  }
}

struct MkEpi {
  int M;
  const int* rows;  // shared-memory copy of the phase's compacted row list
  int* pos;         // [kMaxRows] RoPE position of each compacted row (QKV)
  int* kvslot;      // [kMaxRows] KV-cache slot and row of each compacted row (QKV)
  int* kvrow;
  int nM;           // rows of the next norm phase (residual phases) and their list
  const int* nrows;
  float* xch;    // [16][128]
  float* redv;   // [4][16]
  int* redi;     // [4][16]
  float* rs;     // [kMaxRows] per-row RMSNorm factors of the current phase
  const float* rcos;  // [16][D/2] RoPE cos / sin of the first 16 rows (QKV), staged at phase start
  const float* rsin;
  const float* gnext;  // residual phases: RMSNorm gain of the next norm phase
  bool direct_xn;      // residual phases: the next norm phase runs the same rows in the same order,
                       // so the epilogue writes its B operand straight from the updated h
  int hpre_tile;       // residual phases: tile whose h rows were preloaded into xch (-1: none)
  float gn_pre;        // ... and this thread's next-norm gain on that tile
  // values the epilogue chunks would otherwise load from the step descriptor in global memory
  __nv_bfloat16* kv_base;  // QKV: this layer's KV cache
  size_t kv_cap;
  float* logits;           // LM head: caller's logits or null
  int q, lane, et;
};

// Wait until every 128-feature tile of h has reached `dep`, then compute the RMSNorm factors of
// the phase's rows from the partial sums of squares (fixed order, deterministic).
__device__ bool mk_prepare_rs(const MkParams& p, const MkEpi& e, unsigned long long dep, const MkShared& sh,
                              bool& ready) {
  if (ready) return true;  // once per phase
  ready = true;
  const int nt = p.d / 128;
  bool ok = true;
  for (int t = e.et; dep != 0ull && t < nt && ok; t += 128) ok = mk_wait_flag(&p.hflag[t], dep, sh);
  if (!bar_and(1, 128, ok)) return false;
  for (int j = e.et; j < e.M; j += 128) {
    const int m = e.rows[j];
    float ss = 0.f;
#pragma unroll 8
    for (int t = 0; t < nt; ++t) ss += __ldcg(&p.ssp[static_cast<size_t>(t) * kMaxRows + m]);
    e.rs[j] = rsqrtf(ss / static_cast<float>(p.d) + p.eps);
  }
  named_bar_sync(1, 128);
  return true;
}

// Fused epilogue of one 16-token chunk (tokens ch*16 ..) of output row r of tile t.
// hv (residual phases, optional): h of these 16 rows at this thread's feature, loaded by the caller
// together with the partial sums.
__device__ void mk_epilogue_chunk(const MkParams& p, const MkPhase& ph, const MkEpi& e, int t, int r, int ch,
                                  const float* v, const float* hv = nullptr) {
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
      // rotation factors first (the first 16 rows staged in shared memory, later rows' loads in
      // flight during the exchange of the partner elements)
      const int i = dim & (half - 1);
      float cs[16], sn[16];
      if (j0 == 0) {
#pragma unroll
        for (int jj = 0; jj < 16; ++jj) {
          cs[jj] = e.rcos[jj * half + i];
          sn[jj] = e.rsin[jj * half + i];
        }
      } else {
#pragma unroll
        for (int jj = 0; jj < 16; ++jj) {
          const bool in = j0 + jj < e.M;
          const size_t pe = static_cast<size_t>(in ? e.pos[j0 + jj] : 0) * half + i;
          cs[jj] = in ? __ldg(&p.rope_cos[pe]) : 0.f;
          sn[jj] = in ? __ldg(&p.rope_sin[pe]) : 0.f;
        }
      }
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) e.xch[jj * 128 + r] = val[jj];
      named_bar_sync(1, 128);
      const int pr = r ^ half;
      float rot[16];
#pragma unroll
      for (int jj = 0; jj < 16; ++jj) {
        const float pv = e.xch[jj * 128 + pr];
        rot[jj] = j0 + jj < e.M ? (dim < half ? val[jj] * cs[jj] - pv * sn[jj] : val[jj] * cs[jj] + pv * sn[jj]) : 0.f;
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
        // q in fp16 (11 significant bits), split exactly into bf16 hi + lo by the attention
        reinterpret_cast<__half*>(p.qbuf)[static_cast<size_t>(j) * d + f] = __float2half_rn(val[jj]);
      } else {
        const size_t off = ((static_cast<size_t>(e.kvslot[j]) * 2 + (sec - 1)) * p.H + head) *
                               e.kv_cap +
                           e.kvrow[j];
        e.kv_base[off * D + dim] = __float2bfloat16_rn(val[jj]);
      }
    }
  } else if (ph.kind == kMkO || ph.kind == kMkDown) {
    // residual add, then this tile's partial sum of squares of the updated rows
    const int o = t * 128 + r;
    const float gn = e.direct_xn ? (t == e.hpre_tile ? e.gn_pre : e.gnext[o]) : 0.f;
    float sq[16];
#pragma unroll
    for (int jj = 0; jj < 16; ++jj) {
      const int j = j0 + jj;
      sq[jj] = 0.f;
      if (j < e.M) {
        float* hp = p.h + static_cast<size_t>(e.rows[j]) * p.d + o;
        // h of the CTA's last tile was loaded at phase start (off the critical path)
        const float nv = (t == e.hpre_tile ? e.xch[jj * 128 + r] : hv ? hv[jj] : __ldcg(hp)) + v[jj];
        *hp = nv;
        sq[jj] = nv * nv;
        if (e.direct_xn) store_split(p.xn, p.xs, j, o, nv * gn);
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
          store_split(p.act, p.xs, j, fcol, g / (1.f + expf(-g)) * u);
        }
      }
    }
    named_bar_sync(1, 128);
  } else {  // LM head: logits (optional) and per-tile argmax, lowest index on ties
    const int o = t * 128 + r;
    const bool valid = o < p.V;
    float* logits = e.logits;
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

// Stores of 4 consecutive features (k % 4 == 0) of row j into the split hi/lo layout: they are
// adjacent in the swizzled 64-element rows, so each part is one 8-byte store.
__device__ __forceinline__ void store_split4(__nv_bfloat16* buf, const XsLayout& L, int j, int k, const float* x) {
  uint32_t hi[2], lo[2];
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    hi[i] = pack_bf16(x[2 * i], x[2 * i + 1]);
    const float h0 = __uint_as_float(hi[i] << 16), h1 = __uint_as_float(hi[i] & 0xffff0000u);
    lo[i] = pack_bf16(x[2 * i] - h0, x[2 * i + 1] - h1);
  }
  *reinterpret_cast<uint2*>(buf + xs_elem(L, j, k, 0)) = make_uint2(hi[0], hi[1]);
  *reinterpret_cast<uint2*>(buf + xs_elem(L, j, k, 1)) = make_uint2(lo[0], lo[1]);
}

// Fix-up of tile t from the partials of contributors cf..cl (in that order): warp q takes the
// groups of G rows q, q + 4, ... and each lane 4 adjacent features of all 128, so that the
// partner elements of RoPE and SwiGLU and the reductions over the tile's features (sums of
// squares, argmax) stay within one warp -- no exchange between the warps and no barrier -- and
// every load and store is a 16- or 8-byte vector.  CB contributors' partials per round of loads.
template <int G, int CB>
__device__ void mk_finalize_by_warps(const MkParams& p, const MkPhase& ph, const MkEpi& e, int t, int cf, int cl,
                                     const float* partials, int n_pad) {
  const int lane = e.lane, f0 = 4 * lane;  // features f0 .. f0 + 3 of the tile
  const int n_groups = (e.M + G - 1) / G;
  const bool resid = ph.kind == kMkO || ph.kind == kMkDown;
  float4 gn = make_float4(0.f, 0.f, 0.f, 0.f);
  if (resid && e.direct_xn) gn = *reinterpret_cast<const float4*>(e.gnext + t * 128 + f0);
  for (int grp = e.q; grp < n_groups; grp += 4) {
    {
      const int j0 = grp * G;
      float v[G][4], hv[G][4];
#pragma unroll
      for (int jj = 0; jj < G; ++jj) {
        const bool in = j0 + jj < e.M;
        float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
        if (resid && in) x = __ldcg(reinterpret_cast<const float4*>(p.h + static_cast<size_t>(e.rows[j0 + jj]) * p.d + t * 128 + f0));
        hv[jj][0] = x.x; hv[jj][1] = x.y; hv[jj][2] = x.z; hv[jj][3] = x.w;
        v[jj][0] = v[jj][1] = v[jj][2] = v[jj][3] = 0.f;
      }
      // contributors in order (deterministic sum), CB partials' loads in flight at once
      for (int c0 = cf; c0 <= cl; c0 += CB) {
        float4 a[CB][G];
#pragma unroll
        for (int q = 0; q < CB; ++q) {
          const bool cin = c0 + q <= cl;
          const float* pa = partials + static_cast<size_t>(c0 + q + t) * 128 * n_pad;
#pragma unroll
          for (int jj = 0; jj < G; ++jj)
            a[q][jj] = cin && j0 + jj < e.M ? __ldcg(reinterpret_cast<const float4*>(pa + (j0 + jj) * 128 + f0))
                                            : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int q = 0; q < CB; ++q)
#pragma unroll
          for (int jj = 0; jj < G; ++jj) {
            v[jj][0] += a[q][jj].x;
            v[jj][1] += a[q][jj].y;
            v[jj][2] += a[q][jj].z;
            v[jj][3] += a[q][jj].w;
          }
      }
#pragma unroll
      for (int jj = 0; jj < G; ++jj) {
        const int j = j0 + jj;
        const bool in = j < e.M;  // uniform over the warp
        if (ph.kind == kMkQkv) {
          const int d = p.d, D = p.D, half = D >> 1;
          const int sec = (t * 128) / d;  // q, k or v: one per tile
          const int fs = t * 128 + f0 - sec * d;
          const int head = fs / D, dim0 = fs - head * D;
          const float rsj = in ? e.rs[j] : 0.f;
          float val[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) val[i] = v[jj][i] * rsj;
          if (sec < 2) {  // rotate-half RoPE: the partner feature dim ^ half sits in lane ^ half / 4
            float rot[4];
            const int pos = in ? e.pos[j] : 0;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const float pv = __shfl_xor_sync(0xffffffffu, val[i], half >> 2);
              const int ii = (dim0 + i) & (half - 1);
              const float c = j < 16 ? e.rcos[j * half + ii] : __ldg(&p.rope_cos[static_cast<size_t>(pos) * half + ii]);
              const float sn = j < 16 ? e.rsin[j * half + ii] : __ldg(&p.rope_sin[static_cast<size_t>(pos) * half + ii]);
              rot[i] = dim0 < half ? val[i] * c - pv * sn : val[i] * c + pv * sn;
            }
#pragma unroll
            for (int i = 0; i < 4; ++i) val[i] = rot[i];
          }
          if (in) {
            if (sec == 0) {  // q in fp16 (11 significant bits), split exactly into bf16 hi + lo by the attention
              const uint32_t w0 = pack_f16(val[0], val[1]), w1 = pack_f16(val[2], val[3]);
              *reinterpret_cast<uint2*>(reinterpret_cast<__half*>(p.qbuf) + static_cast<size_t>(j) * d + fs) =
                  make_uint2(w0, w1);
            } else {
              const size_t off = ((static_cast<size_t>(e.kvslot[j]) * 2 + (sec - 1)) * p.H + head) * e.kv_cap + e.kvrow[j];
              *reinterpret_cast<uint2*>(e.kv_base + off * D + dim0) =
                  make_uint2(pack_bf16(val[0], val[1]), pack_bf16(val[2], val[3]));
            }
          }
        } else if (resid) {
          float nv[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) nv[i] = hv[jj][i] + v[jj][i];
          float sq = (nv[0] * nv[0] + nv[1] * nv[1]) + (nv[2] * nv[2] + nv[3] * nv[3]);
#pragma unroll
          for (int off = 16; off > 0; off >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, off);
          if (in) {
            const int m = e.rows[j];
            *reinterpret_cast<float4*>(p.h + static_cast<size_t>(m) * p.d + t * 128 + f0) =
                make_float4(nv[0], nv[1], nv[2], nv[3]);
            if (e.direct_xn) {
              const float xg[4] = {nv[0] * gn.x, nv[1] * gn.y, nv[2] * gn.z, nv[3] * gn.w};
              store_split4(p.xn, p.xs, j, t * 128 + f0, xg);
            }
            if (lane == 0) p.ssp[static_cast<size_t>(t) * kMaxRows + m] = sq;
          }
        } else if (ph.kind == kMkGu) {  // lanes 0-15: gate features, 16-31: the matching up features
          const float rsj = in ? e.rs[j] : 0.f;
          float x[4], act[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            x[i] = v[jj][i] * rsj;
            const float u = __shfl_xor_sync(0xffffffffu, x[i], 16);
            act[i] = x[i] / (1.f + expf(-x[i])) * u;
          }
          if (in && lane < 16) store_split4(p.act, p.xs, j, t * 64 + f0, act);
        } else {  // LM head: logits and the tile's argmax of row j, lowest index on ties
          const float rsj = in ? e.rs[j] : 0.f;
          float bv = -INFINITY;
          int bi = t * 128 + f0;
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const int o = t * 128 + f0 + i;
            const float val = o < p.V && in ? v[jj][i] * rsj : -INFINITY;
            if (o < p.V && in) {
              if (e.logits) e.logits[static_cast<size_t>(e.rows[j]) * p.V + o] = val;
              if (val != val) report(p.status, kStatusCheck);
            }
            if (val > bv) {
              bv = val;
              bi = o;
            }
          }
#pragma unroll
          for (int off = 16; off > 0; off >>= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bv, off);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, off);
            if (ov > bv || (ov == bv && oi < bi)) {
              bv = ov;
              bi = oi;
            }
          }
          if (in && lane == 0) {
            p.amax_val[static_cast<size_t>(t) * kMaxRows + e.rows[j]] = bv;
            p.amax_idx[static_cast<size_t>(t) * kMaxRows + e.rows[j]] = bi;
          }
        }
      }
    }
  }
}

// After a residual phase finalised tile t of h: write the next norm phase's B operand
// bf16(h * g_next) for features [128t, 128t+128) of every row that phase runs, in its compacted
// order (O -> gate/up of the same layer; down -> QKV of the next layer, or the LM head).
__device__ __forceinline__ int mk_next_slot(const MkParams& p, const MkPhase& ph) {
  if (ph.kind == kMkO) return ph.slot;
  return ph.slot + 1 < p.n_act ? ph.slot + 1 : kFinalSlot;
}

__device__ void mk_write_next_xn(const MkParams& p, const PlanDev* pl, const MkPhase& ph, const MkEpi& e, int t,
                                 int r) {
  const int nslot = mk_next_slot(p, ph);
  const float* g = ph.kind == kMkO ? p.g_mlp + static_cast<size_t>(ph.layer) * p.d
                   : nslot != kFinalSlot ? p.g_attn + static_cast<size_t>(pl->act_layer[nslot]) * p.d
                                         : p.g_final;
  const int M = e.nM;
  const int* rows = e.nrows;
  const int f = t * 128 + r;
  const float gf = g[f];
  for (int n0 = 0; n0 < M; n0 += 8) {
    float hv[8];
#pragma unroll
    for (int u = 0; u < 8; ++u)
      hv[u] = n0 + u < M ? __ldcg(&p.h[static_cast<size_t>(rows[n0 + u]) * p.d + f]) : 0.f;
#pragma unroll
    for (int u = 0; u < 8; ++u)
      if (n0 + u < M) store_split(p.xn, p.xs, n0 + u, f, hv[u] * gf);
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

// The attention of QKV slot `slot` in this CTA: its (request, head, split) items round-robin over
// the grid, each run by all 256 threads of the CTA (team thread ttid; the epilogue warps are
// 0..127) in the weight / activation ring, which every role has stopped using when it enters:
// the epilogue warps after the slot's QKV epilogues, the other warps before their O phase.
// Returns false after a failed wait (the kernel is aborting).
template <int D>
__device__ __forceinline__ bool mk_team_attention(const MkParams& p, const AttnParams& ap0, int slot, int ttid,
                                               uint8_t* ring, size_t ring_bytes, float (*sM)[16], float (*sL)[16],
                                               int* s_last, uint64_t* team, uint32_t& team_n, const MkShared& sh) {
  if (!mk_team_sync(team, team_n, sh)) return false;
  const PlanDev* pl = p.plan;
  AttnParams ap = ap0;
  ap.slot = slot;
  const int c = blockIdx.x, G = gridDim.x;
  const int per_req = p.H * p.attn_splits, n_items = p.B * per_req;
  const unsigned long long want = mk_seq(p.seq_base, slot, kMkQkv);
  if (ttid == 0) mk_trace(p, kMkTracePhases * 8 + 2 * slot);
  fence_proxy_async_shared();  // the ring's async-proxy (TMA / MMA) use ends before generic use
  bool ok = true;
  for (int item = c; ok && item < n_items; item += G) {
    const int b = item / per_req;
    const int head = (item - b * per_req) / p.attn_splits;
    const int split = item - b * per_req - head * p.attn_splits;
    if (pl->slot_crow[slot][b] < 0) continue;
    // the Q, K and V tiles of this head (written by the QKV epilogues of this step)
    auto wait_inputs = [&]() -> bool {
      bool good = true;
      if (ttid < 3) {
        const int tile = (ttid * p.d + head * D) / 128;
        good = mk_wait_flag(&p.qkvflag[tile], want, sh);
      }
      return bar_and(2, kMkThreads, good);
    };
    unsigned long long* atr =
        p.trace && slot == 1 ? p.trace + static_cast<size_t>(blockIdx.x) * kMkTraceSlots + kMkTraceAttn : nullptr;
    bool failed = false;
    const bool wrote = attention_item_resident<D, 2, kMkThreads>(ap, split, head, b, ttid, ring, ring_bytes, sM, sL,
                                                                  s_last, atr, wait_inputs, failed, p.attn_plo != 0);
    if (failed) {
      ok = false;
      break;
    }
    if (wrote) {
      named_bar_sync(2, kMkThreads);  // the head's output precedes the flag's release
      if (ttid == 0) st_release_u64(&p.attflag[b * p.H + head], mk_seq(p.seq_base, slot, kMkAtt));
    }
    named_bar_sync(2, kMkThreads);
  }
  if (ttid == 0) mk_trace(p, kMkTracePhases * 8 + 2 * slot + 1);
  fence_proxy_async_shared();  // generic-proxy use of the ring ends before the next TMA writes
  return mk_team_sync(team, team_n, sh) && ok;
}

template <int D>
__global__ void __launch_bounds__(kMkThreads, 1)
    verify_mk_kernel(const MkParams p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int S = p.stages, n_pad = p.n_pad, KPS = p.kps;
  const int XP = p.xs.parts;
  const uint32_t x_bytes = static_cast<uint32_t>(n_pad) * 128u;  // one block of one k-block of the B operand
  const uint32_t sw_bytes = KPS * kMkWBytes, sx_bytes = KPS * XP * x_bytes;
  uint8_t* sW = base;
  uint8_t* sX = sW + static_cast<size_t>(S) * sw_bytes;
  uint8_t* s_attn = sX + static_cast<size_t>(S) * sx_bytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(s_attn + p.attn_extra);
  uint64_t* empty = full + S;
  uint64_t* accf = empty + S;
  uint64_t* acce = accf + kMkMaxAcc;
  uint64_t* team = acce + kMkMaxAcc;  // all 256 threads: entry to / exit from a layer's attention
  int* misc = reinterpret_cast<int*>(team + 1);  // [0] tmem addr, [1] abort, [2..4] bcast, [5] s_last
  float* xch = reinterpret_cast<float*>(misc + 16);
  float* redv = xch + 16 * 128;
  int* redi = reinterpret_cast<int*>(redv + 64);
  float* rs = reinterpret_cast<float*>(redi + 64);
  float (*sM)[16] = reinterpret_cast<float (*)[16]>(rs + kMaxRows);  // [8][16] per attention warp
  float (*sL)[16] = reinterpret_cast<float (*)[16]>(rs + kMaxRows + 128);
  int* s_rows = reinterpret_cast<int*>(rs + kMaxRows + 256);  // [kMaxRows] x 5: rows, pos, kv slot, kv row, next rows
  int* s_pos = s_rows + kMaxRows;
  int* s_kvslot = s_pos + kMaxRows;
  int* s_kvrow = s_kvslot + kMaxRows;
  int* s_nrows = s_kvrow + kMaxRows;
  float* s_rope = reinterpret_cast<float*>(s_nrows + kMaxRows);  // [2][16][64]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int NB = mk_acc_bufs(n_pad);
  const uint32_t ncols = gemm_tmem_cols(n_pad, NB);
  const PlanDev* pl = p.plan;
  const size_t ring_attn_bytes = static_cast<size_t>(s_attn - base) + p.attn_extra;
  MkShared sh;
  sh.abort_s = reinterpret_cast<volatile int*>(misc + 1);
  sh.abort_g = p.abort_word;
  sh.status = p.status;
  sh.limit_ns = p.wait_ns;

  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(&full[i], 2);  // weight TMA arrival + B-operand arrival
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < kMkMaxAcc; ++i) {
      mbar_init(&accf[i], 1);
      mbar_init(&acce[i], 128);
    }
    mbar_init(team, kMkThreads);
    *sh.abort_s = 0;
    fence_mbar_init();
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
  const int n_phases = pl->n_act == p.n_act ? min(4 * p.n_act + 1, p.ph_end) : 0;
  const int ph0 = p.ph_begin;

  // The attention inside this kernel (not with attn_external): every warp joins the team that runs
  // a layer's attention items -- the epilogue warps after the layer's QKV phase, the others before
  // its O phase.
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
  ap.o_xs = p.xs;
  ap.part_o = p.attn_po;
  ap.part_ml = p.attn_pml;
  ap.counters = p.attn_cnt;
  ap.status = p.status;
  uint32_t team_n = 0;
  auto team_attention = [&](int slot) -> bool {
    return mk_team_attention<D>(p, ap, slot, static_cast<int>(threadIdx.x) ^ 128, base, ring_attn_bytes, sM, sL,
                                misc + 5, team, team_n, sh);
  };

  // Roles, all in one loop over the phases: warp 0 lane 0 streams the weights, warp 1 lane 0
  // issues the MMAs, warp 2 loads the B operands, warps 4-7 run the epilogues; at each O phase
  // (inside this kernel's attention) all eight warps first run the layer's attention as one team.
  const uint64_t wpol = l2_policy_evict_first();
  const uint32_t idesc = idesc_bf16_m128(n_pad);
  long long i = 0;  // this role's ring stage counter
  int use = 0;      // this role's accumulator buffer counter
  bool ok = true;
  MkEpi e;
  e.q = warp & 3;
  e.lane = lane;
  e.et = threadIdx.x - 128;
  e.xch = xch;
  e.redv = redv;
  e.redi = redi;
  e.rs = rs;
  e.rcos = s_rope;
  e.rsin = s_rope + 16 * 64;
  const int r = e.q * 32 + lane;
  int* bcast = misc + 2;
  // the weight stages of this CTA's share of a phase: warp 0 lane 0 issues their bulk copies into
  // the ring (it never waits for activations, only for free ring stages)
  auto produce = [&](const MkPhase& ph, int pi) -> bool {
    MkSeg seg = mk_seg(p, ph, c, G);
    const __nv_bfloat16* wl = mk_weights(p, ph);
    int t, k0, k1, j = 0;
    while (seg.next(t, k0, k1)) {
      const bool last_seg = seg.done();
      for (int kc = k0; kc < k1; kc += KPS, ++j) {
        const int nk = min(KPS, k1 - kc);
        const int s = static_cast<int>(i % S);
        if (!mk_wait_bar(&empty[s], static_cast<uint32_t>((i / S) & 1) ^ 1u, sh)) return false;
        if (j == 0) mk_trace(p, pi * 8 + 0);
        if (last_seg && kc + nk == k1) mk_trace(p, pi * 8 + 1);
        mbar_arrive_expect_tx(&full[s], nk * kMkWBytes);
        if (p.w_evict_first)
          bulk_load_hint(sW + static_cast<size_t>(s) * sw_bytes,
                         wl + (static_cast<size_t>(t) * ph.kb + kc) * kTileElems, nk * kMkWBytes, &full[s], wpol);
        else
          bulk_load(sW + static_cast<size_t>(s) * sw_bytes,
                    wl + (static_cast<size_t>(t) * ph.kb + kc) * kTileElems, nk * kMkWBytes, &full[s]);
        ++i;
      }
    }
    return true;
  };
  for (int pi = ph0; ok && pi < n_phases; ++pi) {
    const MkPhase ph = mk_phase(p, pl, pi);
    if (ph.kind == kMkO && !p.attn_external) {
      // this layer's attention: the epilogue warps come after the QKV epilogues (every QKV MMA of
      // this CTA has completed), the other warps before they start the O phase
      const bool t = team_attention(ph.slot);
      ok = warp >= 4 ? bar_and(1, 128, t) : __shfl_sync(0xffffffffu, t, 0);
      if (!ok) break;
    }
    if (warp == 0) {
      // ---------------- weight TMA producer (lane 0): never waits for activations ----------------
      bool good = true;
      if (lane == 0) good = produce(ph, pi);
      ok = __shfl_sync(0xffffffffu, good, 0);
    } else if (warp == 1) {
      // ---------------- MMA issuer (lane 0) ----------------
      if (lane == 0) {
        MkSeg seg = mk_seg(p, ph, c, G);
        int t, k0, k1;
        bool first = true;
        while (ok && seg.next(t, k0, k1)) {
          const int buf = use % NB;
          if (!mk_wait_bar(&acce[buf], static_cast<uint32_t>((use / NB) & 1) ^ 1u, sh)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(buf * n_pad);
          for (int kc = k0; kc < k1; kc += KPS, ++i) {
            const int nk = min(KPS, k1 - kc);
            const int s = static_cast<int>(i % S);
            if (!mk_wait_bar(&full[s], static_cast<uint32_t>((i / S) & 1), sh)) {
              ok = false;
              break;
            }
            tc_fence_after();
            if (first) mk_trace(p, pi * 8 + 4);
            first = false;
            for (int j = 0; j < nk; ++j) {
              const uint32_t a0 = smem_u32(sW + static_cast<size_t>(s) * sw_bytes + j * kMkWBytes);
              const uint32_t b0 = smem_u32(sX + static_cast<size_t>(s) * sx_bytes + j * XP * x_bytes);
              // (branch outside the issue loops: a conditional MMA inside them was measured to
              // slow every stage down)
              if (XP == 1) {
#pragma unroll
                for (int k16 = 0; k16 < 4; ++k16)
                  umma_bf16(d_tmem, sdesc_sw128(a0 + k16 * 32), sdesc_sw128(b0 + k16 * 32), idesc,
                            (kc + j > k0 || k16 > 0) ? 1u : 0u);
              } else {  // the lo block accumulates into the same columns
#pragma unroll
                for (int k16 = 0; k16 < 4; ++k16) {
                  umma_bf16(d_tmem, sdesc_sw128(a0 + k16 * 32), sdesc_sw128(b0 + k16 * 32), idesc,
                            (kc + j > k0 || k16 > 0) ? 1u : 0u);
                  umma_bf16(d_tmem, sdesc_sw128(a0 + k16 * 32), sdesc_sw128(b0 + x_bytes + k16 * 32), idesc, 1u);
                }
              }
            }
            umma_commit(&empty[s]);
          }
          if (!ok) break;
          umma_commit(&accf[buf]);
          if (seg.done()) mk_trace(p, pi * 8 + 5);
          ++use;
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
    } else if (warp == 2) {
      // ---------------- B-operand producer: TMA after the producing tiles are flagged ----------------
      MkSeg seg = mk_seg(p, ph, c, G);
      if (seg.done()) continue;
      // dependency index space of this phase: h tiles, heads, or gate/up tiles
      const unsigned long long* flags;
      unsigned long long want;
      int n_dep;
      if (ph.kind == kMkO) {
        flags = p.attflag;
        want = p.attn_external ? 0ull : mk_seq(p.seq_base, ph.slot, kMkAtt);  // else: an earlier launch
        n_dep = p.H;
      } else if (ph.kind == kMkDown) {
        flags = p.guflag;
        want = mk_seq(p.seq_base, ph.slot, kMkGu);
        n_dep = p.Ft;
      } else {
        flags = p.hflag;
        want = mk_h_dep(p, ph);
        n_dep = p.d / 128;
      }
      const __nv_bfloat16* xsrc = ph.kind == kMkO ? p.obuf : ph.kind == kMkDown ? p.act : p.xn;
      uint32_t ready[8] = {0, 0, 0, 0, 0, 0, 0, 0};  // known-complete dependency indices (<= 256)
      // one flag index is complete when every request that runs the slot has it (attention) or
      // the single flag reached `want`
      auto poll = [&](int x) -> bool {
        if (ph.kind != kMkO) return ld_acquire_u64(&flags[x]) >= want;
        for (int b = 0; b < p.B; ++b)
          if (pl->slot_crow[ph.slot][b] >= 0 && ld_acquire_u64(&flags[b * p.H + x]) < want) return false;
        return true;
      };
      int t, k0, k1;
      bool first = true;
      while (ok && seg.next(t, k0, k1)) {
       const bool last_seg = seg.done();
       for (int kc = k0; ok && kc < k1; kc += KPS, ++i) {
        const int nk = min(KPS, k1 - kc);
        const int s = static_cast<int>(i % S);
        if (lane == 0) ok = mk_wait_bar(&empty[s], static_cast<uint32_t>((i / S) & 1) ^ 1u, sh);
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) break;
        for (int kk = kc; kk < kc + nk; ++kk) {
        const int x = want == 0ull ? -1 : (ph.kind == kMkO ? kk * 64 / p.D : ph.kind == kMkDown ? kk : (kk >> 1));
        if (x >= 0 && !((ready[x >> 5] >> (x & 31)) & 1u)) {
          // poll x .. x+31 at once; then wait (bounded) for x itself if it is not there yet
          const int y = x + lane;
          const bool rdy = y < n_dep && poll(y);
          const uint32_t bal = __ballot_sync(0xffffffffu, rdy);
          __syncwarp();  // memory ordering: lane 0's copy follows the acquire loads of the others
          for (int l = 0; l < 32; ++l)
            if ((bal >> l) & 1u) ready[(x + l) >> 5] |= 1u << ((x + l) & 31);
          if (!(bal & 1u)) {
            bool got = true;
            if (lane == 0) {
              const uint64_t t0 = globaltimer_ns();
              while (!poll(x)) {
                if (mk_aborted(sh)) {
                  got = false;
                  break;
                }
                if (globaltimer_ns() - t0 > sh.limit_ns) {
                  mk_fail(sh);
                  got = false;
                  break;
                }
                __nanosleep(64);
              }
            }
            ok = __shfl_sync(0xffffffffu, got, 0);
            if (!ok) break;
            ready[x >> 5] |= 1u << (x & 31);
          }
        }
        }
        if (!ok) break;
        if (lane == 0) {
          if (first) mk_trace(p, pi * 8 + 2);
          if (last_seg && kc + nk == k1) mk_trace(p, pi * 8 + 3);
          fence_proxy_async_global();
          mbar_arrive_expect_tx(&full[s], nk * XP * x_bytes);
          bulk_load(sX + static_cast<size_t>(s) * sx_bytes, xsrc + static_cast<size_t>(kc) * XP * n_pad * 64, nk * XP * x_bytes,
                    &full[s]);
        }
        first = false;
       }
      }
    } else if (warp >= 4) {
      // ---------------- epilogues ----------------
      MkSeg seg = mk_seg(p, ph, c, G);
      if (seg.done() && ph.kind != kMkQkv) continue;
      // per-phase row metadata in shared memory (loaded while the first accumulator is pending)
      const int rslot = mk_row_slot(ph);
      e.M = pl->slot_M[rslot];
      named_bar_sync(1, 128);  // previous phase's readers of the caches are done
      for (int j = e.et; j < e.M; j += 128) {
        const int m = pl->slot_rows[rslot][j];
        s_rows[j] = m;
        if (ph.kind == kMkQkv) {
          const int b = p.step->row_req[m];
          s_pos[j] = p.step->row_pos[m];
          s_kvslot[j] = p.step->req_slot[b];
          s_kvrow[j] = p.step->req_ctx[b] + (m - p.step->req_rowoff[b]);
        }
      }
      e.direct_xn = false;
      if (ph.kind == kMkO || ph.kind == kMkDown) {
        const int ns = mk_next_slot(p, ph);
        e.nM = pl->slot_M[ns];
        bool same = e.nM == e.M;
        for (int j = e.et; j < e.nM; j += 128) {
          const int m = pl->slot_rows[ns][j];
          s_nrows[j] = m;
          same = same && j < e.M && pl->slot_rows[rslot][j] == m;
        }
        e.direct_xn = bar_and(1, 128, same);
        e.gnext = ph.kind == kMkO ? p.g_mlp + static_cast<size_t>(ph.layer) * p.d
                  : ns != kFinalSlot ? p.g_attn + static_cast<size_t>(pl->act_layer[ns]) * p.d
                                     : p.g_final;
      }
      named_bar_sync(1, 128);
      e.rows = s_rows;
      e.pos = s_pos;
      e.kvslot = s_kvslot;
      e.kvrow = s_kvrow;
      e.nrows = s_nrows;
      e.hpre_tile = -1;
      if ((ph.kind == kMkO || ph.kind == kMkDown) && !seg.done() && e.M <= 16) {
        // h is final for this phase (only this phase's finaliser of a tile writes it): load the
        // rows of the CTA's last tile now, one thread per feature, into xch (unused by residual
        // epilogues), so that finalising that tile -- typically the phase's last -- skips a
        // memory round trip
        const int tl = static_cast<int>((seg.it1 - 1) / ph.kb);  // (residual phases: plain stream-K)
        float hv[16];
#pragma unroll
        for (int jj = 0; jj < 16; ++jj)
          hv[jj] = jj < e.M ? __ldcg(&p.h[static_cast<size_t>(s_rows[jj]) * p.d + tl * 128 + e.q * 32 + lane]) : 0.f;
#pragma unroll
        for (int jj = 0; jj < 16; ++jj) xch[jj * 128 + e.q * 32 + lane] = hv[jj];
        e.hpre_tile = tl;
        e.gn_pre = e.direct_xn ? e.gnext[tl * 128 + e.q * 32 + lane] : 0.f;
      }
      if (ph.kind == kMkQkv) {
        e.kv_base = p.step->kv_layer[ph.layer];
        e.kv_cap = static_cast<size_t>(p.step->kv_cap);
      }
      if (ph.kind == kMkLm) e.logits = p.step->logits;
      if (ph.kind == kMkQkv) {
        // stage the RoPE factors of the first 16 rows; warm L2 with the context keys and values
        // this CTA's attention items will read (they do not depend on this step)
        const int half = D / 2, m16 = e.M < 16 ? e.M : 16;
        for (int x = e.et; x < m16 * half; x += 128) {
          const int j = x / half, i = x - j * half;
          s_rope[j * half + i] = p.rope_cos[static_cast<size_t>(s_pos[j]) * half + i];
          s_rope[16 * 64 + j * half + i] = p.rope_sin[static_cast<size_t>(s_pos[j]) * half + i];
        }
        if (e.et == 0 && !p.attn_external) {
          const int per_req = p.H * p.attn_splits;
          const StepDesc* st = p.step;
          for (int item = c; item < p.B * per_req; item += G) {
            const int b = item / per_req;
            const int head = (item - b * per_req) / p.attn_splits;
            const int split = item - b * per_req - head * p.attn_splits;
            if (pl->slot_crow[ph.slot][b] < 0) continue;
            const int ctx = st->req_ctx[b];
            int k0, k1;
            attn_split_keys(ctx + st->req_nodes[b], p.attn_splits, split, k0, k1);
            k1 = k1 < ctx ? k1 : ctx;
            if (k1 <= k0) continue;
            const size_t cap = static_cast<size_t>(st->kv_cap);
            const __nv_bfloat16* kg =
                st->kv_layer[ph.layer] + ((static_cast<size_t>(st->req_slot[b]) * 2) * p.H + head) * cap * D;
            const uint32_t bytes = static_cast<uint32_t>(k1 - k0) * D * 2;
            bulk_prefetch_l2(kg + static_cast<size_t>(k0) * D, bytes);
            bulk_prefetch_l2(kg + static_cast<size_t>(p.H) * cap * D + static_cast<size_t>(k0) * D, bytes);
          }
        }
        named_bar_sync(1, 128);
      }
      bool rs_ready = false;
      const long long T = seg.T;
      const int geff = seg.geff;
      float* partials = (pi & 1) ? p.partials1 : p.partials0;
      int* counters = p.counters + static_cast<size_t>(ph.kind) * p.max_tiles;
      const bool needs_rs = ph.kind == kMkQkv || ph.kind == kMkGu || ph.kind == kMkLm;
      const unsigned long long hdep = needs_rs ? mk_h_dep(p, ph) : 0ull;
      // the norm factors need only h, which is final before this phase's first accumulator
      if (needs_rs && !mk_prepare_rs(p, e, hdep, sh, rs_ready)) {
        ok = false;
        break;
      }
      int t, k0, k1;
      bool first = true;
      while (ok && seg.next(t, k0, k1)) {
        const int buf = use % NB;
        const bool got = e.et == 0 ? mk_wait_bar(&accf[buf], static_cast<uint32_t>((use / NB) & 1), sh) : true;
        if (!bar_and(1, 128, got)) {
          ok = false;
          break;
        }
        if (e.et == 0 && first) mk_trace(p, pi * 8 + 6);
        first = false;
        tc_fence_after();
        const uint32_t tb = tmem_base + (static_cast<uint32_t>(e.q * 32) << 16) + static_cast<uint32_t>(buf * n_pad);
        const int n_ch = (e.M + 15) >> 4;  // 16-token chunks of the accumulator
        const bool tr_last = e.et == 0 && seg.done();
        if (tr_last) mk_trace(p, kMkTraceSub + pi * 8 + 0);
        bool finalize = false;
        int cf = 0, cl = 0;
        if (k0 == 0 && k1 == ph.kb) {
          if (needs_rs && !mk_prepare_rs(p, e, hdep, sh, rs_ready)) {
            ok = false;
            break;
          }
          for (int ch = 0; ch < n_ch; ++ch) {
            float v[16];
            mk_acc_tokens(tb, ch, p.xs, v);
            mk_epilogue_chunk(p, ph, e, t, r, ch, v);
          }
          tc_fence_before();
          mbar_arrive(&acce[buf]);
          finalize = true;
        } else {
          float* part = partials + static_cast<size_t>(c + t) * 128 * n_pad;
          for (int ch = 0; ch < n_ch; ++ch) {
            float v[16];
            mk_acc_tokens(tb, ch, p.xs, v);
#pragma unroll
            for (int jj = 0; jj < 16; ++jj)
              if (ch * 16 + jj < e.M) __stcg(&part[(ch * 16 + jj) * 128 + r], v[jj]);
          }
          tc_fence_before();
          mbar_arrive(&acce[buf]);
          named_bar_sync(1, 128);  // every thread's partial stores precede the release below
          if (tr_last) mk_trace(p, kMkTraceSub + pi * 8 + 1);
          if (e.et == 0) {
            const int f = mk_cta_of(static_cast<long long>(t) * ph.kb, T, geff);
            const int l = mk_cta_of(static_cast<long long>(t + 1) * ph.kb - 1, T, geff);
            const int old = atom_add_acq_rel_gpu(&counters[t], 1);
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
          if (tr_last) mk_trace(p, kMkTraceSub + pi * 8 + 2);
          if (finalize) {  // (the counter's acquire, then the barrier: the other partials are visible)
            if (needs_rs && !mk_prepare_rs(p, e, hdep, sh, rs_ready)) {
              ok = false;
              break;
            }
            if (tr_last) mk_trace(p, kMkTraceSub + pi * 8 + 3);
            if (e.M <= 8 && cl - cf < 8) {
              // up to 8 rows and 8 contributors: every partial in one round of loads, two rows a warp
              mk_finalize_by_warps<2, 8>(p, ph, e, t, cf, cl, partials, n_pad);
              if (tr_last) mk_trace(p, kMkTraceSub + pi * 8 + 7);
            } else if (e.M > 16) {
              mk_finalize_by_warps<8, 2>(p, ph, e, t, cf, cl, partials, n_pad);
            } else {
              // contributors in order (deterministic sum), four partials' loads in flight at once
              const bool pre_h = (ph.kind == kMkO || ph.kind == kMkDown) && t != e.hpre_tile;
              for (int ch = 0; ch < n_ch; ++ch) {
                float v[16], hv[16];
#pragma unroll
                for (int jj = 0; jj < 16; ++jj) {
                  v[jj] = 0.f;
                  hv[jj] = pre_h && ch * 16 + jj < e.M
                               ? __ldcg(&p.h[static_cast<size_t>(e.rows[ch * 16 + jj]) * p.d + t * 128 + r])
                               : 0.f;
                }
                for (int c0 = cf; c0 <= cl; c0 += 4) {
                  float pv[4][16];
#pragma unroll
                  for (int q = 0; q < 4; ++q) {
                    const bool cin = c0 + q <= cl;
                    const float* pa = partials + static_cast<size_t>(c0 + q + t) * 128 * n_pad;
#pragma unroll
                    for (int jj = 0; jj < 16; ++jj)
                      pv[q][jj] = cin && ch * 16 + jj < e.M ? __ldcg(&pa[(ch * 16 + jj) * 128 + r]) : 0.f;
                  }
#pragma unroll
                  for (int q = 0; q < 4; ++q)
#pragma unroll
                    for (int jj = 0; jj < 16; ++jj) v[jj] += pv[q][jj];
                }
                mk_epilogue_chunk(p, ph, e, t, r, ch, v, pre_h ? hv : nullptr);
              }
            }
            if (tr_last) mk_trace(p, kMkTraceSub + pi * 8 + 4);
          }
        }
        if (finalize) {
          unsigned long long* flag = mk_tile_flag(p, ph.kind, t);
          if ((ph.kind == kMkO || ph.kind == kMkDown) && !e.direct_xn) {
            named_bar_sync(1, 128);  // h of this tile is final for every row of the phase
            mk_write_next_xn(p, pl, ph, e, t, r);
          }
          if (tr_last) mk_trace(p, kMkTraceSub + pi * 8 + 5);
          named_bar_sync(1, 128);  // the tile's outputs precede the flag's release
          if (tr_last) mk_trace(p, kMkTraceSub + pi * 8 + 6);
          // (fault injection for the timeout path: the first h tile of the first layer's down
          // phase is never flagged, so its consumers' bounded waits run out)
          const bool withheld = p.withhold_flag && ph.kind == kMkDown && ph.slot == 0 && t == 0;
          if (flag && e.et == 0 && !withheld) st_release_u64(flag, mk_seq(p.seq_base, ph.slot, ph.kind));
        }
        if (e.et == 0 && seg.done()) mk_trace(p, pi * 8 + 7);
        ++use;
      }
    }
  }
  if (warp == 0 && lane == 0 && (!ok || *sh.abort_s)) {  // let weight tiles in flight land before the CTA exits
    const uint64_t t0 = globaltimer_ns();
    while (globaltimer_ns() - t0 < 50000) {
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

size_t mk_trace_slots() { return kMkTraceSlots; }

size_t mk_smem_bytes(int n_pad, int parts, int stages, int head_dim, int kps, size_t attn_extra) {
  return 1024 + static_cast<size_t>(stages) * kps * (kMkWBytes + static_cast<size_t>(n_pad) * parts * 128) +
         attn_extra + static_cast<size_t>(2 * stages + 2 * kMkMaxAcc + 1) * 8 + 64 + 16 * 128 * 4 +
         64 * 4 * 2 + kMaxRows * 4 + 256 * 4 + 5 * kMaxRows * 4 + 2 * 16 * 64 * 4 + 64;
}

cudaError_t mk_prepare() {
  cudaError_t e = cudaFuncSetAttribute(verify_mk_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, 232448);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(verify_mk_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, 232448);
  return e;
}

cudaError_t launch_verify_mk(const MkParams& p, int grid, size_t smem, cudaStream_t s) {
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
  if (p.D == 64) return cudaLaunchKernelEx(&cfg, verify_mk_kernel<64>, p);
  if (p.D == 128) return cudaLaunchKernelEx(&cfg, verify_mk_kernel<128>, p);
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
