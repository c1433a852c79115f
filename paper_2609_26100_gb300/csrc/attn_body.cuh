// Device-side body of the split-KV draft-block attention (see attention.cu for the
// mathematics); shared by the standalone attention kernel and the persistent verify kernel.
#pragma once

#include "internal.h"

namespace tss {

constexpr int kAttnThreads = 128;
constexpr int kKeyTile = 64;

template <int D>
constexpr int attn_ld() {
  return D + 8;  // padded smem row (bf16 elements): conflict-free ldmatrix
}

__host__ __device__ inline size_t attn_qlo_bytes(int head_dim) {
  return static_cast<size_t>(kNarrowNodes) * (head_dim + 8) * 2;  // lo parts of q
}

// The separate kernel's wide variant (blocks of up to 128 rows): Q of 128 rows, and its lo part.
__host__ __device__ inline size_t attn_wide_smem_bytes(int head_dim) {
  const size_t ld = head_dim + 8;
  return static_cast<size_t>(2 * kMaxNodes + 4 * kKeyTile) * ld * 2;
}
__host__ __device__ inline size_t attn_smem_bytes_impl(int head_dim) {
  const int ld = head_dim + 8;
  return static_cast<size_t>(kNarrowNodes + 4 * kKeyTile) * ld * 2;  // Q + double-buffered K and V
}

// Keys [k0, k1) that split `split` of n_splits covers in a block of T keys (whole 64-key tiles,
// the last split possibly shorter or empty).
__host__ __device__ inline void attn_split_keys(int T, int n_splits, int split, int& k0, int& k1) {
  const int n_tiles = (T + kKeyTile - 1) / kKeyTile;
  const int per = (n_tiles + n_splits - 1) / n_splits;
  const int t0 = split * per;
  const int t1 = t0 + per < n_tiles ? t0 + per : n_tiles;
  k0 = t0 * kKeyTile;
  k1 = t1 * kKeyTile < T ? t1 * kKeyTile : T;
}

// Per-item geometry shared by the two item variants below.
template <int D>
struct AttnItem {
  const __nv_bfloat16* Kg;  // this (request, head)'s keys / values in the cache: [cap][D]
  const __nv_bfloat16* Vg;
  int crow, N, ctx, T, t0, t1, mt, wm, wk, ksplit, kpw, g, tq, warp, lane;
  unsigned long long anc0, anc1;
  const unsigned long long* anc_hi;  // blocks of more than 64 rows: ancestor bits of block rows 64..127 by row
};

// Fills `it` for thread `tid` of a team of NT threads; false when the request does not run this
// layer or the item is out of range.
// NB: block rows the item's buffers hold (64, or 128 for the separate kernel's wide variant).
template <int D, int NT = kAttnThreads, int NB = kNarrowNodes>
__device__ __forceinline__ bool attn_item_setup(const AttnParams& p, int split, int head, int b, int tid,
                                                AttnItem<D>& it) {
  const StepDesc* st = p.step;
  const PlanDev* pl = p.plan;
  if (b >= st->B || p.slot >= pl->n_act) return false;
  it.crow = pl->slot_crow[p.slot][b];
  if (it.crow < 0) return false;  // request skips this layer: no KV read, no output
  const int layer = pl->act_layer[p.slot];
  const int H = p.n_heads;
  it.N = st->req_nodes[b];
  it.ctx = st->req_ctx[b];
  it.T = it.ctx + it.N;
  const int row0 = st->req_rowoff[b];
  const size_t cap = static_cast<size_t>(st->kv_cap);
  const int n_tiles = (it.T + kKeyTile - 1) / kKeyTile;
  const int per = (n_tiles + p.n_splits - 1) / p.n_splits;
  it.t0 = split * per;
  it.t1 = min(n_tiles, it.t0 + per);
  it.Kg = st->kv_layer[layer] + ((static_cast<size_t>(st->req_slot[b]) * 2 + 0) * H + head) * cap * D;
  it.Vg = it.Kg + static_cast<size_t>(H) * cap * D;
  it.warp = tid >> 5;
  it.lane = tid & 31;
  it.mt = it.N <= 16 ? 1 : (it.N <= 32 ? 2 : (NB > kNarrowNodes && it.N > kNarrowNodes ? 8 : 4));  // 16-row query tiles
  it.ksplit = NT / 32 / it.mt;  // warps sharing one query tile
  it.wm = it.warp % it.mt;
  it.wk = it.warp / it.mt;
  it.kpw = kKeyTile / it.ksplit;  // keys of each tile this warp scores (tile-sliced variant)
  it.g = it.lane >> 2;
  it.tq = it.lane & 3;
  const int qr0 = it.wm * 16 + it.g, qr1 = qr0 + 8;
  it.anc0 = qr0 < it.N ? st->row_anc[row0 + qr0] : 0ull;
  it.anc1 = qr1 < it.N ? st->row_anc[row0 + qr1] : 0ull;
  if constexpr (NB > kNarrowNodes) it.anc_hi = st->row_anc_hi + row0;
  return true;
}

// Q rows of the request into sQ [16 * mt][LD] (rows >= N are zero); cp.async, not committed.
template <int D, int NT = kAttnThreads>
__device__ __forceinline__ void attn_load_q(const AttnParams& p, const AttnItem<D>& it, int head, int tid,
                                            __nv_bfloat16* sQ) {
  constexpr int LD = attn_ld<D>(), C8 = D / 8;
  for (int idx = tid; idx < 16 * it.mt * C8; idx += NT) {
    const int row = idx / C8, c8 = idx - row * C8;
    __nv_bfloat16* dst = sQ + row * LD + c8 * 8;
    if (row < it.N) {
      cp_async16(dst, p.q + static_cast<size_t>(it.crow + row) * p.d_model + head * D + c8 * 8, 16);
    } else {
      *reinterpret_cast<uint4*>(dst) = make_uint4(0, 0, 0, 0);
    }
  }
}

// Keys and values of one 64-key tile into sK / sV [kKeyTile][LD]; keys past the block are
// zero-filled.  cp.async, not committed.
template <int D, int NT = kAttnThreads>
__device__ __forceinline__ void attn_load_tile(const AttnItem<D>& it, int tile, int tid, __nv_bfloat16* sK,
                                               __nv_bfloat16* sV) {
  constexpr int LD = attn_ld<D>(), C8 = D / 8;
  for (int idx = tid; idx < kKeyTile * C8; idx += NT) {
    const int kr = idx / C8, c8 = idx - kr * C8;
    const int key = tile * kKeyTile + kr;
    const int bytes = key < it.T ? 16 : 0;
    const size_t src = static_cast<size_t>(key < it.T ? key : 0) * D + c8 * 8;
    cp_async16(sK + kr * LD + c8 * 8, it.Kg + src, bytes);
    cp_async16(sV + kr * LD + c8 * 8, it.Vg + src, bytes);
  }
}

// Online-softmax state of one warp: O accumulators of its two query rows (per lane fragment),
// running max and sum in log2 units, and the Q fragments.
template <int D>
struct AttnAcc {
  float o[D / 8][4];
  float m0, m1, l0, l1;
  uint32_t qf[D / 16][4];
  uint32_t qlo[D / 16][4];  // lo parts of q (bf16) when the scores use q = hi + lo
};

template <int D>
__device__ __forceinline__ void attn_acc_init(AttnAcc<D>& a) {
#pragma unroll
  for (int i = 0; i < D / 8; ++i) a.o[i][0] = a.o[i][1] = a.o[i][2] = a.o[i][3] = 0.f;
  a.m0 = a.m1 = -INFINITY;
  a.l0 = a.l1 = 0.f;
}

template <int D>
__device__ __forceinline__ void attn_load_qfrag(const AttnItem<D>& it, const __nv_bfloat16* sQ, AttnAcc<D>& a) {
  constexpr int LD = attn_ld<D>();
#pragma unroll
  for (int ks = 0; ks < D / 16; ++ks)
    ldmatrix_x4(a.qf[ks], sQ + (it.wm * 16 + (it.lane & 15)) * LD + ks * 16 + (it.lane >> 4) * 8);
}

// q arrives in fp16 (11 significant bits) and is split exactly into two bf16 parts: hi in place
// of q, lo into sQlo (rows of the warps' query tiles).
template <int D, int NT = kAttnThreads>
__device__ __forceinline__ void attn_split_q(const AttnItem<D>& it, __nv_bfloat16* sQ, __nv_bfloat16* sQlo, int tid) {
  constexpr int LD = attn_ld<D>(), C2 = D / 2;
  for (int idx = tid; idx < 16 * it.mt * C2; idx += NT) {
    const int row = idx / C2, c2 = idx - row * C2;
    uint32_t* qw = reinterpret_cast<uint32_t*>(sQ + row * LD) + c2;
    const __half2 hq = *reinterpret_cast<const __half2*>(qw);
    const float2 f = __half22float2(hq);
    const uint32_t hi = pack_bf16(f.x, f.y);
    const float hx = __uint_as_float(hi << 16), hy = __uint_as_float(hi & 0xffff0000u);
    *qw = hi;
    reinterpret_cast<uint32_t*>(sQlo + row * LD)[c2] = pack_bf16(f.x - hx, f.y - hy);
  }
}

template <int D>
__device__ __forceinline__ void attn_load_qfrag_hilo(const AttnItem<D>& it, const __nv_bfloat16* sQ,
                                                     const __nv_bfloat16* sQlo, AttnAcc<D>& a) {
  constexpr int LD = attn_ld<D>();
  attn_load_qfrag<D>(it, sQ, a);
#pragma unroll
  for (int ks = 0; ks < D / 16; ++ks)
    ldmatrix_x4(a.qlo[ks], sQlo + (it.wm * 16 + (it.lane & 15)) * LD + ks * 16 + (it.lane >> 4) * 8);
}

// One online-softmax update over up to four 16-key blocks of this warp (kp / vp: their first K
// and V rows in shared memory, key0: the key index of their first row): scores, context /
// ancestor mask, rescale, P.V.  The blocks' score MMAs are independent, so a group of blocks
// from several resident tiles keeps the tensor pipe busier than one block at a time.
// QK16: fp16 score MMAs, q in fp16 (a.qf) and each bf16 key fragment converted to fp16 in
// registers (exact for |k| in [6.1e-5, 65504]).  PLO: P.V with P as two bf16 parts,
// hi = bf16(p) and lo = bf16(p - hi), both multiplied by the bf16 values (else P in bf16).
// QLO: bf16 scores with q as two bf16 parts (a.qf hi, a.qlo lo), keys as stored.
// WIDE: blocks of more than 64 rows (the ancestor bits of block rows 64..127 come from it.anc_hi).
template <int D, bool QK16 = false, bool PLO = false, bool QLO = false, bool WIDE = false>
__device__ __forceinline__ void attn_blocks_step(const AttnItem<D>& it, const __nv_bfloat16* const (&kp)[4],
                                                 const __nv_bfloat16* const (&vp)[4], const int (&key0)[4], int n,
                                                 float scale_log2, AttnAcc<D>& a) {
  constexpr int LD = attn_ld<D>();
  const int lane = it.lane;
  float s[8][4];
#pragma unroll
  for (int nt = 0; nt < 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
  for (int ks = 0; ks < D / 16; ++ks) {
#pragma unroll
    for (int np = 0; np < 4; ++np) {
      if (np < n) {
        uint32_t kb4[4];
        ldmatrix_x4(kb4, kp[np] + ((lane & 7) + ((lane >> 4) << 3)) * LD + ks * 16 + ((lane >> 3) & 1) * 8);
        if (QK16) {
#pragma unroll
          for (int j = 0; j < 4; ++j) kb4[j] = bf16x2_to_f16x2(kb4[j]);
          mma_f16_16816(s[2 * np], a.qf[ks], kb4);
          mma_f16_16816(s[2 * np + 1], a.qf[ks], kb4 + 2);
        } else if (QLO) {
          mma_bf16_16816(s[2 * np], a.qf[ks], kb4);
          mma_bf16_16816(s[2 * np + 1], a.qf[ks], kb4 + 2);
          mma_bf16_16816(s[2 * np], a.qlo[ks], kb4);
          mma_bf16_16816(s[2 * np + 1], a.qlo[ks], kb4 + 2);
        } else {
          mma_bf16_16816(s[2 * np], a.qf[ks], kb4);
          mma_bf16_16816(s[2 * np + 1], a.qf[ks], kb4 + 2);
        }
      }
    }
  }
  // scale to log2 units and apply the context / ancestor mask
  float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
  for (int nt = 0; nt < 8; ++nt) {
    if (nt < 2 * n) {
      const int kb0 = key0[nt >> 1] + (nt & 1) * 8;
      const bool need_mask = key0[nt >> 1] + 16 > it.ctx;
#pragma unroll
      for (int e2 = 0; e2 < 4; ++e2) {
        float val = s[nt][e2] * scale_log2;
        if (need_mask) {
          const int key = kb0 + it.tq * 2 + (e2 & 1);
          if constexpr (WIDE) {
            const int j = key - it.ctx;  // block row of the key
            const int qr = it.wm * 16 + it.g + (e2 < 2 ? 0 : 8);
            const unsigned long long anc = j < 64 ? (e2 < 2 ? it.anc0 : it.anc1) : (qr < it.N ? it.anc_hi[qr] : 0ull);
            if (key >= it.T || (j >= 0 && !((anc >> (j & 63)) & 1ull))) val = -INFINITY;
          } else {
            const unsigned long long anc = e2 < 2 ? it.anc0 : it.anc1;
            if (key >= it.T || (key >= it.ctx && !((anc >> (key - it.ctx)) & 1ull))) val = -INFINITY;
          }
        }
        s[nt][e2] = val;
      }
      mx0 = fmaxf(mx0, fmaxf(s[nt][0], s[nt][1]));
      mx1 = fmaxf(mx1, fmaxf(s[nt][2], s[nt][3]));
    }
  }
  mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
  mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
  mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
  mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
  const float mn0 = fmaxf(a.m0, mx0), mn1 = fmaxf(a.m1, mx1);
  const float base0 = mn0 == -INFINITY ? 0.f : mn0;
  const float base1 = mn1 == -INFINITY ? 0.f : mn1;
  const float al0 = exp2f(a.m0 - base0), al1 = exp2f(a.m1 - base1);
  a.m0 = mn0;
  a.m1 = mn1;
  float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
  for (int nt = 0; nt < 8; ++nt) {
    if (nt < 2 * n) {
      s[nt][0] = exp2f(s[nt][0] - base0);
      s[nt][1] = exp2f(s[nt][1] - base0);
      s[nt][2] = exp2f(s[nt][2] - base1);
      s[nt][3] = exp2f(s[nt][3] - base1);
      rs0 += s[nt][0] + s[nt][1];
      rs1 += s[nt][2] + s[nt][3];
    }
  }
  a.l0 = a.l0 * al0 + rs0;
  a.l1 = a.l1 * al1 + rs1;
#pragma unroll
  for (int dt = 0; dt < D / 8; ++dt) {
    a.o[dt][0] *= al0;
    a.o[dt][1] *= al0;
    a.o[dt][2] *= al1;
    a.o[dt][3] *= al1;
  }
#pragma unroll
  for (int kc = 0; kc < 4; ++kc) {
    if (kc < n) {
      uint32_t pa[4], pl[4];
      pa[0] = pack_bf16(s[2 * kc][0], s[2 * kc][1]);
      pa[1] = pack_bf16(s[2 * kc][2], s[2 * kc][3]);
      pa[2] = pack_bf16(s[2 * kc + 1][0], s[2 * kc + 1][1]);
      pa[3] = pack_bf16(s[2 * kc + 1][2], s[2 * kc + 1][3]);
      if (PLO) {
        // residuals of the rounding: p - float(bf16(p)), packed the same way
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float x0 = (i < 2 ? s[2 * kc][2 * (i & 1)] : s[2 * kc + 1][2 * (i & 1)]);
          const float x1 = (i < 2 ? s[2 * kc][2 * (i & 1) + 1] : s[2 * kc + 1][2 * (i & 1) + 1]);
          const float h0 = __uint_as_float(pa[i] << 16), h1 = __uint_as_float(pa[i] & 0xffff0000u);
          pl[i] = pack_bf16(x0 - h0, x1 - h1);
        }
      }
#pragma unroll
      for (int dp = 0; dp < D / 16; ++dp) {
        uint32_t vb[4];
        ldmatrix_x4_trans(vb, vp[kc] + ((lane & 7) + (((lane >> 3) & 1) << 3)) * LD + dp * 16 + (lane >> 4) * 8);
        mma_bf16_16816(a.o[2 * dp], pa, vb);
        mma_bf16_16816(a.o[2 * dp + 1], pa, vb + 2);
        if (PLO) {
          mma_bf16_16816(a.o[2 * dp], pl, vb);
          mma_bf16_16816(a.o[2 * dp + 1], pl, vb + 2);
        }
      }
    }
  }
}

// This warp's keys of one resident 64-key tile (K / V buffers sK, sV).
template <int D, bool QK16 = false, bool PLO = false, bool QLO = false, bool WIDE = false>
__device__ __forceinline__ void attn_tile_step(const AttnItem<D>& it, int tile, const __nv_bfloat16* sK,
                                               const __nv_bfloat16* sV, float scale_log2, AttnAcc<D>& a) {
  constexpr int LD = attn_ld<D>();
  const int kbase = it.wk * it.kpw;
  const __nv_bfloat16* kp[4];
  const __nv_bfloat16* vp[4];
  int key0[4];
#pragma unroll
  for (int np = 0; np < 4; ++np) {
    kp[np] = sK + (kbase + np * 16) * LD;
    vp[np] = sV + (kbase + np * 16) * LD;
    key0[np] = tile * kKeyTile + kbase + np * 16;
  }
  attn_blocks_step<D, QK16, PLO, QLO, WIDE>(it, kp, vp, key0, it.kpw / 16, scale_log2, a);
}

// Weighted sum over the splits of every output element of a (request, head): each thread takes
// kU elements per round with the partial outputs of all (<= kS) splits loaded together; the first
// round's loads are issued before `weights()` (which computes wgt) so that they overlap.
template <int D, int NT, int kU, int kS, typename Weights, typename Put, int NB = kNarrowNodes>
__device__ __forceinline__ void attn_merge_rounds(const AttnParams& p, size_t ph, int N, int ns, int tid,
                                                  const float* wgt, Weights weights, Put put) {
  float po[kU][kS];
  auto load = [&](int idx0) {
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int idx = idx0 + u * NT;
      const int i = idx / D, dd = idx - i * D;
#pragma unroll
      for (int sp = 0; sp < kS; ++sp)
        po[u][sp] = idx < N * D && sp < ns ? __ldcg(&p.part_o[((ph + sp) * NB + i) * D + dd]) : 0.f;
    }
  };
  load(tid);
  weights();
  for (int idx0 = tid; idx0 < N * D; idx0 += kU * NT) {
    if (idx0 != tid) load(idx0);
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int idx = idx0 + u * NT;
      if (idx >= N * D) continue;
      const float* w = wgt + (idx / D) * ns;
      float o = 0.f;
#pragma unroll
      for (int sp = 0; sp < kS; ++sp)
        if (sp < ns) o += w[sp] * po[u][sp];
      put(idx, o);
    }
  }
}

// Merge the warps that share a query tile through shared memory (sO: [NT / 32][16][D] floats, any
// free 16-byte-aligned buffer of NT / 4 KiB for D = 128; sM, sL: [NT / 32][16]), then write this split's result: the
// normalised output when there is one split, else the partial, and the last split of
// (request, head) merges all partials in split order.  Returns true on the call that wrote the
// final output rows.  `stamp(k)` records diagnostics (k = 9, 2, 3, 4 in that order).
// kFastMerge: the merge's loads in one round (attn_merge_rounds), used by the persistent
// kernel; the standalone kernel keeps the plain loop, which measured faster there.
template <int D, int BAR, int NT, bool kFastMerge, typename Stamp, int NB = kNarrowNodes>
__device__ __forceinline__ bool attn_finish(const AttnParams& p, const AttnItem<D>& it, AttnAcc<D>& a, int split,
                                            int head, int b, int tid, float* sO, float (*sM)[16], float (*sL)[16],
                                            int* s_last, Stamp stamp) {
  const int H = p.n_heads, d = p.d_model;
  constexpr int NW = NT / 32;
  const int N = it.N, crow = it.crow, mt = it.mt, warp = it.warp, g = it.g, tq = it.tq;
  a.l0 += __shfl_xor_sync(0xffffffffu, a.l0, 1);
  a.l0 += __shfl_xor_sync(0xffffffffu, a.l0, 2);
  a.l1 += __shfl_xor_sync(0xffffffffu, a.l1, 1);
  a.l1 += __shfl_xor_sync(0xffffffffu, a.l1, 2);

  named_bar_sync(BAR, NT);
#pragma unroll
  for (int dt = 0; dt < D / 8; ++dt) {
    const int col = dt * 8 + tq * 2;
    sO[(warp * 16 + g) * D + col] = a.o[dt][0];
    sO[(warp * 16 + g) * D + col + 1] = a.o[dt][1];
    sO[(warp * 16 + g + 8) * D + col] = a.o[dt][2];
    sO[(warp * 16 + g + 8) * D + col + 1] = a.o[dt][3];
  }
  if (tq == 0) {
    sM[warp][g] = a.m0;
    sM[warp][g + 8] = a.m1;
    sL[warp][g] = a.l0;
    sL[warp][g + 8] = a.l1;
  }
  named_bar_sync(BAR, NT);
  stamp(9);

  const size_t ph = (static_cast<size_t>(b) * H + head) * p.n_splits;
  // Per query row (one thread each): the warps' common max M, their weights 2^(m_w - M) (written
  // over sM) and the merged sum L (over sL of the row's first warp); then every output element
  // is a plain weighted sum of the warps' O, the loads of several elements in flight.
  for (int i = tid; i < N; i += NT) {
    const int wt = i >> 4, rr = i & 15;
    float M = -INFINITY;
    for (int w = wt; w < NW; w += mt) M = fmaxf(M, sM[w][rr]);
    const float base = M == -INFINITY ? 0.f : M;
    float L = 0.f;
    for (int w = wt; w < NW; w += mt) {
      const float f = exp2f(sM[w][rr] - base);
      L += f * sL[w][rr];
      sM[w][rr] = f;
    }
    sL[wt][rr] = L;
    if (p.n_splits == 1) {
      if (!(L > 0.f)) report(p.status, kStatusCheck);
    } else {
      const size_t pi = (ph + split) * NB + i;
      __stcg(&p.part_ml[pi * 2 + 0], M);
      __stcg(&p.part_ml[pi * 2 + 1], L);
    }
  }
  named_bar_sync(BAR, NT);
#pragma unroll 4
  for (int idx = tid; idx < N * D; idx += NT) {
    const int i = idx / D, dd = idx - i * D;
    const int wt = i >> 4, rr = i & 15;
    float O = 0.f;
    for (int w = wt; w < NW; w += mt) O += sM[w][rr] * sO[(w * 16 + rr) * D + dd];
    if (p.n_splits == 1) {
      const float L = sL[wt][rr];
      const float val = L > 0.f ? O / L : 0.f;
      if (p.o_xs.rows)
        store_split(p.o, p.o_xs, crow + i, head * D + dd, val);
      else
        p.o[static_cast<size_t>(crow + i) * d + head * D + dd] = __float2bfloat16_rn(val);
    } else {
      __stcg(&p.part_o[((ph + split) * NB + i) * D + dd], O);
    }
  }
  if (p.n_splits == 1) return true;
  stamp(2);

  // Last CTA of (request, head) merges the splits in order.
  named_bar_sync(BAR, NT);  // every thread's partial stores precede the release below
  if (tid == 0) {
    int* cnt = p.counters + static_cast<size_t>(b) * H + head;
    const int old = atom_add_acq_rel_gpu(cnt, 1);
    *s_last = old == p.n_splits - 1;
    if (*s_last) atomicExch(cnt, 0);
  }
  named_bar_sync(BAR, NT);
  stamp(3);
  if (!*s_last) return false;  // (the counter's acquire, then the barrier: the partials are visible)
  if (kFastMerge) {
    // Merge weights per (row, split) -- w = 2^(m_s - M) / L with L = sum 2^(m_s - M) l_s, in split
    // order -- and the weighted sum of the splits' O for every output element.  The (m, l) pairs go
    // to shared memory (sO is free again) while the first elements' partial outputs are already in
    // flight, so that the merge of a small block costs one round of loads.
    const int ns = p.n_splits;
    float* wgt = sO;                          // [N][ns]
    float* sml = sO + NB * kMaxSplits;  // [N][ns] x (m, l)
    for (int x = tid; x < N * ns; x += NT) {
      const int i = x / ns, sp = x - i * ns;
      const size_t pi = (ph + sp) * NB + i;
      sml[2 * x] = __ldcg(&p.part_ml[pi * 2]);
      sml[2 * x + 1] = __ldcg(&p.part_ml[pi * 2 + 1]);
    }
    auto weights = [&]() {
      named_bar_sync(BAR, NT);
      for (int i = tid; i < N; i += NT) {
        float M = -INFINITY;
        for (int sp = 0; sp < ns; ++sp) M = fmaxf(M, sml[2 * (i * ns + sp)]);
        const float base = M == -INFINITY ? 0.f : M;
        float L = 0.f;
        for (int sp = 0; sp < ns; ++sp) {
          const float f = exp2f(sml[2 * (i * ns + sp)] - base);
          L += f * sml[2 * (i * ns + sp) + 1];
          wgt[i * ns + sp] = f;
        }
        if (!(L > 0.f)) report(p.status, kStatusCheck);
        const float inv = L > 0.f ? 1.f / L : 0.f;
        for (int sp = 0; sp < ns; ++sp) wgt[i * ns + sp] *= inv;
      }
      named_bar_sync(BAR, NT);
    };
    auto put = [&](int idx, float val) {
      const int i = idx / D, dd = idx - i * D;
      if (p.o_xs.rows)
        store_split(p.o, p.o_xs, crow + i, head * D + dd, val);
      else
        p.o[static_cast<size_t>(crow + i) * d + head * D + dd] = __float2bfloat16_rn(val);
    };
    if (ns <= 4)
      attn_merge_rounds<D, NT, 8, 4, decltype(weights), decltype(put), NB>(p, ph, N, ns, tid, wgt, weights, put);
    else if (ns <= 8)
      attn_merge_rounds<D, NT, 4, 8, decltype(weights), decltype(put), NB>(p, ph, N, ns, tid, wgt, weights, put);
    else
      attn_merge_rounds<D, NT, 2, 16, decltype(weights), decltype(put), NB>(p, ph, N, ns, tid, wgt, weights, put);
  } else {
    // Merge weights per (row, split) first -- w = 2^(m_s - M) / L with L = sum 2^(m_s - M) l_s, in
    // split order -- into shared memory (sO is free again), then every output element is a
    // weighted sum of the splits' O, several elements' loads in flight per thread.
    float* wgt = sO;  // [N][n_splits]
    const int ns = p.n_splits;
    for (int i = tid; i < N; i += NT) {
      float M = -INFINITY;
      for (int sp = 0; sp < ns; ++sp) M = fmaxf(M, __ldcg(&p.part_ml[((ph + sp) * NB + i) * 2]));
      const float base = M == -INFINITY ? 0.f : M;
      float L = 0.f;
      for (int sp = 0; sp < ns; ++sp) {
        const size_t pi = (ph + sp) * NB + i;
        const float f = exp2f(__ldcg(&p.part_ml[pi * 2]) - base);
        L += f * __ldcg(&p.part_ml[pi * 2 + 1]);
        wgt[i * ns + sp] = f;
      }
      if (!(L > 0.f)) report(p.status, kStatusCheck);
      const float inv = L > 0.f ? 1.f / L : 0.f;
      for (int sp = 0; sp < ns; ++sp) wgt[i * ns + sp] *= inv;
    }
    named_bar_sync(BAR, NT);
    constexpr int kU = 4;  // output elements per thread with their loads in flight together
    for (int idx0 = tid; idx0 < N * D; idx0 += kU * NT) {
      float O[kU];
  #pragma unroll
      for (int u = 0; u < kU; ++u) O[u] = 0.f;
      for (int sp = 0; sp < ns; ++sp) {
        float po[kU];
  #pragma unroll
        for (int u = 0; u < kU; ++u) {
          const int idx = idx0 + u * NT;
          const int i = idx / D, dd = idx - i * D;
          po[u] = idx < N * D ? __ldcg(&p.part_o[((ph + sp) * NB + i) * D + dd]) : 0.f;
        }
  #pragma unroll
        for (int u = 0; u < kU; ++u) {
          const int idx = idx0 + u * NT;
          if (idx < N * D) O[u] += wgt[(idx / D) * ns + sp] * po[u];
        }
      }
  #pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int idx = idx0 + u * NT;
        if (idx >= N * D) continue;
        const int i = idx / D, dd = idx - i * D;
        if (p.o_xs.rows)
          store_split(p.o, p.o_xs, crow + i, head * D + dd, O[u]);
        else
          p.o[static_cast<size_t>(crow + i) * d + head * D + dd] = __float2bfloat16_rn(O[u]);
      }
    }
  }
  stamp(4);
  return true;
}

// One work item (split, head, request) run by 128 threads (tid 0..127) that synchronise with
// named barrier BAR, streaming its key tiles through a double buffer.  smem: attn_smem_bytes(D)
// bytes, 16-byte aligned.  Returns true on the call that wrote the final output rows of
// (request, head) (the only split, or the last split to finish, which merges the others in
// split order).  P16: the persistent path's operands and precision (q arrives in fp16 and is split
// once into bf16 hi/lo parts for the score MMAs, so the bf16 keys need no conversion; P as hi/lo
// bf16 parts in P.V; output split hi/lo); else all bf16.  With P16 the kernel needs
// attn_smem_bytes(D) + attn_qlo_bytes(D) of shared memory.
// NB / NT: block rows the buffers hold and threads of the item -- 64 and 128, or the wide variant
// for blocks of up to 128 rows, 128 and 256 (eight query tiles, one warp each).
template <int D, int BAR, bool P16 = false, int NB = kNarrowNodes, int NT = kAttnThreads>
__device__ bool attention_item(const AttnParams& p, int split, int head, int b, int tid, uint8_t* smem,
                               float (*sM)[16], float (*sL)[16], int* s_last) {
  constexpr int LD = attn_ld<D>();
  __nv_bfloat16* sQ = reinterpret_cast<__nv_bfloat16*>(smem);  // [NB][LD]
  __nv_bfloat16* sK = sQ + NB * LD;                              // [2][kKeyTile][LD]
  __nv_bfloat16* sV = sK + 2 * kKeyTile * LD;                    // [2][kKeyTile][LD]
  AttnItem<D> it;
  if (!attn_item_setup<D, NT, NB>(p, split, head, b, tid, it)) return false;
  attn_load_q<D, NT>(p, it, head, tid, sQ);
  if (it.t0 < it.t1) attn_load_tile<D, NT>(it, it.t0, tid, sK, sV);
  cp_async_commit();
  AttnAcc<D> a;
  attn_acc_init<D>(a);
  for (int tile = it.t0; tile < it.t1; ++tile) {
    const int buf = (tile - it.t0) & 1;
    if (tile + 1 < it.t1)
      attn_load_tile<D, NT>(it, tile + 1, tid, sK + (buf ^ 1) * kKeyTile * LD, sV + (buf ^ 1) * kKeyTile * LD);
    cp_async_commit();
    cp_async_wait<1>();
    named_bar_sync(BAR, NT);
    if (tile == it.t0) {
      if (P16) {
        __nv_bfloat16* sQlo = sV + 2 * kKeyTile * LD;
        attn_split_q<D, NT>(it, sQ, sQlo, tid);
        named_bar_sync(BAR, NT);
        attn_load_qfrag_hilo<D>(it, sQ, sQlo, a);
      } else {
        attn_load_qfrag<D>(it, sQ, a);
      }
    }
    attn_tile_step<D, false, P16, P16, (NB > kNarrowNodes)>(it, tile, sK + buf * kKeyTile * LD, sV + buf * kKeyTile * LD,
                                                          p.scale_log2, a);
    named_bar_sync(BAR, NT);
  }
  cp_async_wait<0>();
  auto no_stamp = [](int) {};
  return attn_finish<D, BAR, NT, false, decltype(no_stamp), NB>(p, it, a, split, head, b, tid, reinterpret_cast<float*>(sK),
                                                             sM, sL, s_last, no_stamp);
}

// Tiles of K and V that attention_item_resident keeps resident in `smem_bytes` of shared memory.
__host__ __device__ inline int attn_resident_tiles(int head_dim, size_t smem_bytes) {
  const size_t ld = head_dim + 8, q = static_cast<size_t>(kNarrowNodes) * ld * 2, tile = 2ull * kKeyTile * ld * 2;
  return smem_bytes > q ? static_cast<int>((smem_bytes - q) / tile) : 0;
}

// The same work item with all of the split's key tiles resident at once (in rounds of
// attn_resident_tiles(D, smem_bytes) tiles when they do not all fit): loads of tiles that hold
// only context keys (which this step does not write) are issued first, then `wait_inputs()`
// waits for the step's own Q/K/V rows, then Q and the remaining tiles are loaded.  One memory
// round trip per round instead of one per tile.  The scores are fp16 MMAs (q arrives in fp16, the
// keys are converted in registers).  Run by a team of NT threads (tid < NT); each warp scores
// every (NT / 32 / query tiles)-th 16-key block of a round.  Needs smem_bytes >= the Q buffer +
// 1 tile and the NT / 4 KiB merge buffer (D = 128) to fit behind Q.  If wait_inputs() fails,
// drains its copies and returns false without output.
template <int D, int BAR, int NT, typename Wait>
__device__ bool attention_item_resident(const AttnParams& p, int split, int head, int b, int tid, uint8_t* smem,
                                        size_t smem_bytes, float (*sM)[16], float (*sL)[16], int* s_last,
                                        unsigned long long* trace, Wait wait_inputs, bool& failed, bool plo = true) {
  constexpr int LD = attn_ld<D>();
  auto stamp = [&](int k) {
    if (trace && tid == 0) trace[k] = globaltimer_ns();
  };
  failed = false;
  __nv_bfloat16* sQ = reinterpret_cast<__nv_bfloat16*>(smem);  // [kNarrowNodes][LD] (q in fp16)
  __nv_bfloat16* sKV = sQ + kNarrowNodes * LD;                   // per tile slot: K [kKeyTile][LD], V [kKeyTile][LD]
  const int R = attn_resident_tiles(D, smem_bytes);
  AttnItem<D> it;
  const bool run = attn_item_setup<D, NT>(p, split, head, b, tid, it);
  if (!run || R < 1) {
    failed = !wait_inputs();
    return false;
  }
  auto tile_k = [&](int slot) { return sKV + slot * 2 * kKeyTile * LD; };
  auto tile_v = [&](int slot) { return sKV + (slot * 2 + 1) * kKeyTile * LD; };
  auto load_round = [&](int r0, int r1, int slot0, bool ctx_only) {
    for (int tile = r0; tile < r1; ++tile)
      if (!ctx_only || (tile + 1) * kKeyTile <= it.ctx)
        attn_load_tile<D, NT>(it, tile, tid, tile_k(slot0 + tile - r0), tile_v(slot0 + tile - r0));
  };
  AttnAcc<D> a;
  attn_acc_init<D>(a);
  // this warp's 16-key blocks of tiles [r0, r1) held from slot0 on -- every ksplit-th block of
  // the round, starting at wk -- four per softmax update
  auto score_round = [&](int r0, int r1, int slot0) {
    constexpr int kBlocks = kKeyTile / 16;  // 16-key blocks per tile
    const int nall = (r1 - r0) * kBlocks;
    const int nb = nall > it.wk ? (nall - it.wk + it.ksplit - 1) / it.ksplit : 0;
    for (int q0 = 0; q0 < nb; q0 += 4) {
      const __nv_bfloat16* kp[4];
      const __nv_bfloat16* vp[4];
      int key0[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int gb = it.wk + min(q0 + j, nb - 1) * it.ksplit;
        const int tl = gb / kBlocks, np = gb - tl * kBlocks;
        kp[j] = tile_k(slot0 + tl) + np * 16 * LD;
        vp[j] = tile_v(slot0 + tl) + np * 16 * LD;
        key0[j] = (r0 + tl) * kKeyTile + np * 16;
      }
      if (plo)
        attn_blocks_step<D, true, true>(it, kp, vp, key0, min(4, nb - q0), p.scale_log2, a);
      else
        attn_blocks_step<D, true, false>(it, kp, vp, key0, min(4, nb - q0), p.scale_log2, a);
    }
  };
  const int nt = it.t1 - it.t0;
  if (nt <= R) {
    // one round: the context tiles (which this step does not write) are requested first, the
    // Q rows and the block's own tiles once the step's QKV flags are set
    load_round(it.t0, it.t1, 0, true);
    cp_async_commit();
    if (!wait_inputs()) {
      cp_async_wait<0>();
      failed = true;
      return false;
    }
    attn_load_q<D, NT>(p, it, head, tid, sQ);
    for (int tile = it.t0; tile < it.t1; ++tile)
      if ((tile + 1) * kKeyTile > it.ctx) attn_load_tile<D, NT>(it, tile, tid, tile_k(tile - it.t0), tile_v(tile - it.t0));
    cp_async_commit();
    cp_async_wait<0>();
    named_bar_sync(BAR, NT);
    stamp(0);
    attn_load_qfrag<D>(it, sQ, a);
    score_round(it.t0, it.t1, 0);
    named_bar_sync(BAR, NT);
  } else {
    // Rounds of H tiles through two halves of the resident space: the next round's copies are in
    // flight while this round is scored.  Round 0 holds only context tiles (the block's own keys
    // are in the last two tiles at most, and nt > R >= 2H).
    const int nbuf = R >= 2 ? 2 : 1;
    const int H = R / nbuf;
    const int nr = (nt + H - 1) / H;
    load_round(it.t0, min(it.t1, it.t0 + H), 0, false);
    cp_async_commit();
    if (!wait_inputs()) {
      cp_async_wait<0>();
      failed = true;
      return false;
    }
    attn_load_q<D, NT>(p, it, head, tid, sQ);
    cp_async_commit();
    for (int r = 0; r < nr; ++r) {
      const int r0 = it.t0 + r * H, r1 = min(it.t1, r0 + H);
      const int slot0 = (r % nbuf) * H;
      if (nbuf == 1 && r > 0) {
        load_round(r0, r1, 0, false);
        cp_async_commit();
      }
      if (nbuf == 2 && r + 1 < nr) {
        const int n0 = r0 + H;
        load_round(n0, min(it.t1, n0 + H), ((r + 1) % 2) * H, false);
        cp_async_commit();
        cp_async_wait<1>();
      } else {
        cp_async_wait<0>();
      }
      named_bar_sync(BAR, NT);
      if (r == 0) {
        stamp(0);
        attn_load_qfrag<D>(it, sQ, a);
      }
      score_round(r0, r1, slot0);
      named_bar_sync(BAR, NT);  // this half is reloaded by the round after next
    }
  }
  stamp(1);
  if (trace && it.lane == 0 && it.warp < 4) trace[5 + it.warp] = globaltimer_ns();
  return attn_finish<D, BAR, NT, true>(p, it, a, split, head, b, tid, reinterpret_cast<float*>(sKV), sM, sL, s_last, stamp);
}

}  // namespace tss
