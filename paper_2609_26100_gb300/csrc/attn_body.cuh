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

__host__ __device__ inline size_t attn_smem_bytes_impl(int head_dim) {
  const int ld = head_dim + 8;
  return static_cast<size_t>(kMaxNodes + 4 * kKeyTile) * ld * 2;  // Q + double-buffered K and V
}

// One work item (split, head, request) run by 128 threads (tid 0..127) that synchronise with
// named barrier BAR.  smem: attn_smem_bytes(D) bytes, 16-byte aligned.  Returns true on the
// call that wrote the final output rows of (request, head) (the only split, or the last split to
// finish, which merges the others in split order).
template <int D, int BAR>
__device__ bool attention_item(const AttnParams& p, int split, int head, int b, int tid, uint8_t* smem,
                               float (*sM)[16], float (*sL)[16], int* s_last) {
  constexpr int LD = attn_ld<D>();
  __nv_bfloat16* sQ = reinterpret_cast<__nv_bfloat16*>(smem);  // [kMaxNodes][LD]
  __nv_bfloat16* sK = sQ + kMaxNodes * LD;                       // [2][kKeyTile][LD]
  __nv_bfloat16* sV = sK + 2 * kKeyTile * LD;                    // [2][kKeyTile][LD]
  const StepDesc* st = p.step;
  const PlanDev* pl = p.plan;
  if (b >= st->B || p.slot >= pl->n_act) return false;
  const int crow = pl->slot_crow[p.slot][b];
  if (crow < 0) return false;  // request skips this layer: no KV read, no output
  const int layer = pl->act_layer[p.slot];
  const int H = p.n_heads, d = p.d_model;
  const int N = st->req_nodes[b], ctx = st->req_ctx[b], T = ctx + N;
  const int row0 = st->req_rowoff[b];
  const size_t cap = static_cast<size_t>(st->kv_cap);
  const int n_tiles = (T + kKeyTile - 1) / kKeyTile;
  const int per = (n_tiles + p.n_splits - 1) / p.n_splits;
  const int t0 = split * per;
  const int t1 = min(n_tiles, t0 + per);
  const __nv_bfloat16* Kg =
      st->kv_layer[layer] + ((static_cast<size_t>(st->req_slot[b]) * 2 + 0) * H + head) * cap * D;
  const __nv_bfloat16* Vg = Kg + static_cast<size_t>(H) * cap * D;

  const int warp = tid >> 5, lane = tid & 31;
  const int mt = N <= 16 ? 1 : (N <= 32 ? 2 : 4);  // 16-row query tiles
  const int ksplit = 4 / mt;                        // warps sharing one query tile
  const int wm = warp % mt, wk = warp / mt;
  const int kpw = kKeyTile / ksplit;  // keys of each tile this warp scores
  const int g = lane >> 2, tq = lane & 3;
  const int qr0 = wm * 16 + g, qr1 = qr0 + 8;
  const unsigned long long anc0 = qr0 < N ? st->row_anc[row0 + qr0] : 0ull;
  const unsigned long long anc1 = qr1 < N ? st->row_anc[row0 + qr1] : 0ull;

  // Q rows of the request (rows >= N are zero).
  constexpr int C8 = D / 8;
  for (int idx = tid; idx < 16 * mt * C8; idx += kAttnThreads) {
    const int row = idx / C8, c8 = idx - row * C8;
    __nv_bfloat16* dst = sQ + row * LD + c8 * 8;
    if (row < N) {
      cp_async16(dst, p.q + static_cast<size_t>(crow + row) * d + head * D + c8 * 8, 16);
    } else {
      *reinterpret_cast<uint4*>(dst) = make_uint4(0, 0, 0, 0);
    }
  }
  auto load_tile = [&](int tile, int buf) {
    for (int idx = tid; idx < kKeyTile * C8; idx += kAttnThreads) {
      const int kr = idx / C8, c8 = idx - kr * C8;
      const int key = tile * kKeyTile + kr;
      const int bytes = key < T ? 16 : 0;  // keys past the block are zero-filled
      const size_t src = static_cast<size_t>(key < T ? key : 0) * D + c8 * 8;
      cp_async16(sK + (buf * kKeyTile + kr) * LD + c8 * 8, Kg + src, bytes);
      cp_async16(sV + (buf * kKeyTile + kr) * LD + c8 * 8, Vg + src, bytes);
    }
  };
  if (t0 < t1) load_tile(t0, 0);
  cp_async_commit();

  float o[D / 8][4];
#pragma unroll
  for (int i = 0; i < D / 8; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  uint32_t qf[D / 16][4];

  for (int tile = t0; tile < t1; ++tile) {
    const int buf = (tile - t0) & 1;
    if (tile + 1 < t1) load_tile(tile + 1, buf ^ 1);
    cp_async_commit();
    cp_async_wait<1>();
    named_bar_sync(BAR, kAttnThreads);
    if (tile == t0) {
#pragma unroll
      for (int ks = 0; ks < D / 16; ++ks)
        ldmatrix_x4(qf[ks], sQ + (wm * 16 + (lane & 15)) * LD + ks * 16 + (lane >> 4) * 8);
    }
    const int kbase = wk * kpw;
    const __nv_bfloat16* tK = sK + (buf * kKeyTile + kbase) * LD;
    const __nv_bfloat16* tV = sV + (buf * kKeyTile + kbase) * LD;
    float s[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
    const int npairs = kpw / 16;
#pragma unroll
    for (int np = 0; np < 4; ++np) {
      if (np < npairs) {
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
          uint32_t kb4[4];
          ldmatrix_x4(kb4, tK + (np * 16 + (lane & 7) + ((lane >> 4) << 3)) * LD + ks * 16 + ((lane >> 3) & 1) * 8);
          mma_bf16_16816(s[2 * np], qf[ks], kb4);
          mma_bf16_16816(s[2 * np + 1], qf[ks], kb4 + 2);
        }
      }
    }
    // scale to log2 units and apply the context / ancestor mask
    const int key0 = tile * kKeyTile + kbase;
    const bool need_mask = tile * kKeyTile + kKeyTile > ctx;
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      if (nt < 2 * npairs) {
#pragma unroll
        for (int e2 = 0; e2 < 4; ++e2) {
          float val = s[nt][e2] * p.scale_log2;
          if (need_mask) {
            const int key = key0 + nt * 8 + tq * 2 + (e2 & 1);
            const unsigned long long anc = e2 < 2 ? anc0 : anc1;
            if (key >= T || (key >= ctx && !((anc >> (key - ctx)) & 1ull))) val = -INFINITY;
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
    const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
    const float base0 = mn0 == -INFINITY ? 0.f : mn0;
    const float base1 = mn1 == -INFINITY ? 0.f : mn1;
    const float al0 = exp2f(m0 - base0), al1 = exp2f(m1 - base1);
    m0 = mn0;
    m1 = mn1;
    float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
    for (int nt = 0; nt < 8; ++nt) {
      if (nt < 2 * npairs) {
        s[nt][0] = exp2f(s[nt][0] - base0);
        s[nt][1] = exp2f(s[nt][1] - base0);
        s[nt][2] = exp2f(s[nt][2] - base1);
        s[nt][3] = exp2f(s[nt][3] - base1);
        rs0 += s[nt][0] + s[nt][1];
        rs1 += s[nt][2] + s[nt][3];
      }
    }
    l0 = l0 * al0 + rs0;
    l1 = l1 * al1 + rs1;
#pragma unroll
    for (int dt = 0; dt < D / 8; ++dt) {
      o[dt][0] *= al0;
      o[dt][1] *= al0;
      o[dt][2] *= al1;
      o[dt][3] *= al1;
    }
#pragma unroll
    for (int kc = 0; kc < 4; ++kc) {
      if (kc < npairs) {
        uint32_t a[4];
        a[0] = pack_bf16(s[2 * kc][0], s[2 * kc][1]);
        a[1] = pack_bf16(s[2 * kc][2], s[2 * kc][3]);
        a[2] = pack_bf16(s[2 * kc + 1][0], s[2 * kc + 1][1]);
        a[3] = pack_bf16(s[2 * kc + 1][2], s[2 * kc + 1][3]);
#pragma unroll
        for (int dp = 0; dp < D / 16; ++dp) {
          uint32_t vb[4];
          ldmatrix_x4_trans(vb, tV + (kc * 16 + (lane & 7) + (((lane >> 3) & 1) << 3)) * LD + dp * 16 + (lane >> 4) * 8);
          mma_bf16_16816(o[2 * dp], a, vb);
          mma_bf16_16816(o[2 * dp + 1], a, vb + 2);
        }
      }
    }
    named_bar_sync(BAR, kAttnThreads);
  }
  cp_async_wait<0>();

  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);

  // Merge the warps that share a query tile (different key subsets) through shared memory.
  named_bar_sync(BAR, kAttnThreads);
  float* sO = reinterpret_cast<float*>(sK);  // [4][16][D] (K/V buffers are free now)
#pragma unroll
  for (int dt = 0; dt < D / 8; ++dt) {
    const int col = dt * 8 + tq * 2;
    sO[(warp * 16 + g) * D + col] = o[dt][0];
    sO[(warp * 16 + g) * D + col + 1] = o[dt][1];
    sO[(warp * 16 + g + 8) * D + col] = o[dt][2];
    sO[(warp * 16 + g + 8) * D + col + 1] = o[dt][3];
  }
  if (tq == 0) {
    sM[warp][g] = m0;
    sM[warp][g + 8] = m1;
    sL[warp][g] = l0;
    sL[warp][g + 8] = l1;
  }
  named_bar_sync(BAR, kAttnThreads);

  const size_t ph = (static_cast<size_t>(b) * H + head) * p.n_splits;
  for (int idx = tid; idx < N * D; idx += kAttnThreads) {
    const int i = idx / D, dd = idx - i * D;
    const int wt = i >> 4, rr = i & 15;
    float M = -INFINITY;
    for (int w = wt; w < 4; w += mt) M = fmaxf(M, sM[w][rr]);
    const float base = M == -INFINITY ? 0.f : M;
    float L = 0.f, O = 0.f;
    for (int w = wt; w < 4; w += mt) {
      const float f = exp2f(sM[w][rr] - base);
      L += f * sL[w][rr];
      O += f * sO[(w * 16 + rr) * D + dd];
    }
    if (p.n_splits == 1) {
      if (!(L > 0.f)) report(p.status, kStatusCheck);
      const float val = L > 0.f ? O / L : 0.f;
      p.o[static_cast<size_t>(crow + i) * d + head * D + dd] = __float2bfloat16_rn(val);
    } else {
      const size_t pi = (ph + split) * kMaxNodes + i;
      __stcg(&p.part_o[pi * D + dd], O);
      if (dd == 0) {
        __stcg(&p.part_ml[pi * 2 + 0], M);
        __stcg(&p.part_ml[pi * 2 + 1], L);
      }
    }
  }
  if (p.n_splits == 1) return true;

  // Last CTA of (request, head) merges the splits in order.
  __threadfence();
  named_bar_sync(BAR, kAttnThreads);
  if (tid == 0) {
    int* cnt = p.counters + static_cast<size_t>(b) * H + head;
    const int old = atomicAdd(cnt, 1);
    *s_last = old == p.n_splits - 1;
    if (*s_last) atomicExch(cnt, 0);
  }
  named_bar_sync(BAR, kAttnThreads);
  if (!*s_last) return false;
  __threadfence();
  for (int idx = tid; idx < N * D; idx += kAttnThreads) {
    const int i = idx / D, dd = idx - i * D;
    float M = -INFINITY;
    for (int sp = 0; sp < p.n_splits; ++sp) M = fmaxf(M, __ldcg(&p.part_ml[((ph + sp) * kMaxNodes + i) * 2]));
    const float base = M == -INFINITY ? 0.f : M;
    float L = 0.f, O = 0.f;
    for (int sp = 0; sp < p.n_splits; ++sp) {
      const size_t pi = (ph + sp) * kMaxNodes + i;
      const float f = exp2f(__ldcg(&p.part_ml[pi * 2]) - base);
      L += f * __ldcg(&p.part_ml[pi * 2 + 1]);
      O += f * __ldcg(&p.part_o[pi * D + dd]);
    }
    if (!(L > 0.f)) report(p.status, kStatusCheck);
    p.o[static_cast<size_t>(crow + i) * d + head * D + dd] = __float2bfloat16_rn(L > 0.f ? O / L : 0.f);
  }
  return true;
}

}  // namespace tss
