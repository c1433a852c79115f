// Split-KV attention of short draft blocks on the 5th-generation tensor cores (tcgen05).
//
// The same operation as attention.cu (App. "Models": rotary multi-head attention of a LLaMA
// block; the draft block is scored in parallel, Sec. "Problem Formulation"): for request b,
// head h and block row q,
//   o_q = softmax_j(q_q . k_j / sqrt(D)) v_j over every context key j < ctx_len and every block
//   key ctx_len + t for which block row t is row q itself or one of its ancestors,
// for blocks of at most 16 rows and head_dim 128.  With so few query rows the keys take the
// 128-row (M) side of the MMA:
//   S^T [128 keys x NQ]  = K [128 keys x D] . Qop^T        (A: K tile, K-major, from TMA)
//   O^T [D x NQ]        += V^T [D x 128 keys] . Pop^T      (A: V tile read MN-major)
// with S^T and O^T in tensor memory.  Operands in two bf16 parts (fp16 q of the persistent
// plan split exactly into hi + lo, and the softmax weights P as hi + lo) stack the parts as rows
// 0-15 and 16-31 of one NQ = 32-row operand, so one MMA per k-step yields both products in
// separate accumulator columns, added in fp32 when read; single-part operands use NQ = 16.
// One thread per key turns its lane of S^T into weights; the running maximum of each query row
// is raised only when a tile's score exceeds it by more than 2^8 (the weights stay finite; the
// sums and O are rescaled then), so a typical tile needs no reduction across keys.
//
// Work split: the (request, head) items of the requests that run this layer, each cut into
// 128-key tiles, are laid end to end and cut into min(grid, tiles) equal ranges, one per CTA
// (one CTA per SM).  A CTA streams its range through two three-slot TMA rings -- keys, released
// as soon as their score product completes, and values, released after P.V -- and produces one
// result per item it covers: the output itself when it holds the whole item, else a partial
// (O, max, sum) that the last CTA to finish the item merges with the others in CTA order.
// Roles (320 threads): warps 0-3 softmax (warp w: TMEM lanes 32w..32w+31 = keys), warps 4-7
// epilogue (the same lanes of O^T = head dimensions; double-buffered O so the next item's P.V
// proceeds meanwhile), warp 8 the TMA producer, warp 9 the MMA issuer.  Every wait is bounded;
// on expiry the kernel records a timeout, drains its copies and MMAs and returns.
#include "internal.h"

namespace tss {

namespace {

constexpr int kTcKeys = 128;    // keys per tile (MMA M of the score product)
constexpr int kTcRows = 16;     // query rows of a block
constexpr int kTcStages = 3;    // slots of each of the K and V rings
constexpr int kTcD = 128;       // head dimension
constexpr int kTcThreads = 320;
constexpr uint32_t kBox = kTcKeys * 64 * 2;   // one 128-key x 64-column swizzled box: 16 KiB
constexpr uint32_t kSlotBytes = 2 * kBox;     // one tile's K (or V): both 64-column boxes
constexpr uint32_t kOpRows = 32;              // operand rows: part hi in rows 0-15, lo in 16-31
constexpr uint32_t kOpBytes = kOpRows * 128;  // one 64-column block of an operand: 4 KiB
constexpr uint32_t kQBytes = 2 * kOpBytes;    // Q operand: 128 columns
constexpr uint32_t kPBytes = 2 * kOpBytes;    // P operand: 128 keys
constexpr uint32_t kTmemCols = 128;           // S^T x 2 (cols 0-63), O^T x 2 (cols 64-127), 32 each
constexpr uint32_t kOCol = 64;
constexpr float kRaise = 8.f;                 // log2 headroom before the running max is raised

struct TcShared {
  uint64_t kfull[kTcStages], kempty[kTcStages], vfull[kTcStages], vempty[kTcStages];
  uint64_t s_full[2], s_free[2], p_full[2], p_free[2], q_full[2];
  uint64_t o_full[2], o_free[2], h_full[2], h_free[2], drain;
  uint32_t tmem;
  int abort;
  int last;
  int cum[kMaxBatch + 1];   // prefix sums of the (request, head) tiles over the requests
  float red[4][kTcRows];    // softmax: per-warp column maxima
  float hm[2][kTcRows];     // softmax -> epilogue: running maxima of an item's part
  float hl[2][4][kTcRows];  // ... and the per-warp sums of its weights
};

__host__ __device__ inline size_t tc_dyn_smem() {
  return static_cast<size_t>(2 * kTcStages) * kSlotBytes + 2 * kQBytes + 2 * kPBytes + 1024;
}

// Descriptor of an MN-major operand in 128-byte-swizzled atoms of 64 elements along M (or N):
// atoms `lbo` bytes apart, 8-row groups along K 1024 bytes apart.
__device__ __forceinline__ uint64_t sdesc_sw128_mn(uint32_t saddr, uint32_t lbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>(1024 >> 4) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}

// Byte offset of element (row r, column k) of a 32-row operand in K-major 128-byte swizzle:
// 64-column blocks of kOpBytes, rows of 128 B, 16-byte chunks permuted by the row.
__device__ __forceinline__ uint32_t op_off(int r, int k) {
  return static_cast<uint32_t>((k >> 6) * kOpBytes + r * 128 + ((((k & 63) >> 3) ^ (r & 7)) << 4) + (k & 7) * 2);
}

// OR of v over the 128 threads of named barrier ID (which it also synchronises).
template <int ID>
__device__ __forceinline__ bool bar_or(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 q, %1, 0;\n\t"
      "bar.red.or.pred p, %2, 128, q;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(r)
      : "r"(v ? 1u : 0u), "n"(ID)
      : "memory");
  return r != 0;
}

constexpr int kBarSoftmax = 1, kBarEpi = 2;

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const float* v) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
      "%16};" ::"r"(taddr),
      "f"(v[0]), "f"(v[1]), "f"(v[2]), "f"(v[3]), "f"(v[4]), "f"(v[5]), "f"(v[6]), "f"(v[7]), "f"(v[8]), "f"(v[9]),
      "f"(v[10]), "f"(v[11]), "f"(v[12]), "f"(v[13]), "f"(v[14]), "f"(v[15])
      : "memory");
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// Wait for a phase that an already-issued copy or MMA will complete, whatever the abort state
// (used before the kernel returns so that nothing writes shared or tensor memory afterwards).
__device__ __forceinline__ void mbar_drain(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait(bar, parity))
    if (globaltimer_ns() - t0 > kWaitLimitNs) return;
}

// The CTA (of C) whose range holds global tile g of T: ranges are [c T / C, (c + 1) T / C).
__device__ __forceinline__ int tc_cta_of(long long g, long long T, int C) {
  return static_cast<int>(((g + 1) * C - 1) / T);
}

// Cursor over a CTA's tiles in the global order (request, head, key tile).
struct TcCursor {
  int b, h, kt, nt;  // nt: tiles of each head of request b
  __device__ void start(const TcShared& sh, int B, int H, long long g) {
    b = 0;
    while (b + 1 < B && sh.cum[b + 1] <= g) ++b;
    nt = (sh.cum[b + 1] - sh.cum[b]) / H;
    const int r = static_cast<int>(g - sh.cum[b]);
    h = r / nt;
    kt = r - h * nt;
  }
  __device__ void next(const TcShared& sh, int B, int H) {
    if (++kt < nt) return;
    kt = 0;
    if (++h < H) return;
    h = 0;
    do {
      ++b;
    } while (b < B && sh.cum[b + 1] == sh.cum[b]);
    if (b < B) nt = (sh.cum[b + 1] - sh.cum[b]) / H;
  }
};

// Q rows of (request b, head h) as the B operand of the score product: rows >= N zero, 128
// columns, K-major 128-byte swizzle.  P16: q arrives in fp16 and is split exactly into bf16 hi
// (rows 0-15) + lo (rows 16-31); else q is bf16 (rows 0-15).
// Each of 128 threads holds two 16-byte chunks (8 columns of one row): tc_load_q reads them
// from the q rows, tc_store_q writes them (split into parts) into an operand buffer.
__device__ __forceinline__ void tc_load_q(const AttnTcParams& p, int crow, int N, int h, int tid, uint4 (&raw)[2]) {
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int x = tid + 128 * i, r = x >> 4, c8 = x & 15;
    raw[i] = make_uint4(0, 0, 0, 0);
    if (r < N) raw[i] = *reinterpret_cast<const uint4*>(p.q + static_cast<size_t>(crow + r) * p.d_model + h * kTcD + c8 * 8);
  }
}

template <bool P16>
__device__ __forceinline__ void tc_store_q(uint8_t* qb, int tid, const uint4 (&rawq)[2]) {
#pragma unroll
  for (int i2 = 0; i2 < 2; ++i2) {
    const int x = tid + 128 * i2, r = x >> 4, c8 = x & 15;
    const uint4 raw = rawq[i2];
    if (P16) {
      const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
      uint32_t hi[4], lo[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&w[i]));
        hi[i] = pack_bf16(f.x, f.y);
        const float hx = __uint_as_float(hi[i] << 16), hy = __uint_as_float(hi[i] & 0xffff0000u);
        lo[i] = pack_bf16(f.x - hx, f.y - hy);
      }
      *reinterpret_cast<uint4*>(qb + op_off(r, c8 * 8)) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
      *reinterpret_cast<uint4*>(qb + op_off(kTcRows + r, c8 * 8)) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
    } else {
      *reinterpret_cast<uint4*>(qb + op_off(r, c8 * 8)) = raw;
    }
  }
}

template <bool P16>
__device__ __forceinline__ void tc_write_q(const AttnTcParams& p, int crow, int N, int h, uint8_t* qb, int tid) {
  uint4 raw[2];
  tc_load_q(p, crow, N, h, tid, raw);
  tc_store_q<P16>(qb, tid, raw);
}

__device__ __forceinline__ void tc_store_out(const AttnTcParams& p, int row, int col, float v) {
  if (p.o_xs.rows)
    store_split(p.o, p.o_xs, row, col, v);
  else
    p.o[static_cast<size_t>(row) * p.d_model + col] = __float2bfloat16_rn(v);
}

// NQ columns of a 32-lane TMEM block (thread i: lane i) to or from v[NQ]
template <int NQ>
__device__ __forceinline__ void tmem_ld_nq(uint32_t taddr, float* v) {
  tmem_ld16(taddr, v);
  if (NQ == 32) tmem_ld16(taddr + 16, v + 16);
}
template <int NQ>
__device__ __forceinline__ void tmem_st_nq(uint32_t taddr, const float* v) {
  tmem_st16(taddr, v);
  if (NQ == 32) tmem_st16(taddr + 16, v + 16);
}

}  // namespace

// Softmax: warps 0-3, thread k owns key row k of every tile (TMEM lane k of S^T).  Per tile:
// scores -> weights P (both parts) into the P operand; at the end of each item's part, its
// running maxima and weight sums go to the epilogue warps.
template <bool P16>
__device__ __forceinline__ void tc_softmax(const AttnTcParams& p, TcShared& sh, uint32_t tm, uint8_t* qbuf,
                                           uint8_t* pbuf, uint8_t* vring, int n, long long g0, int tid, int warp,
                                           int lane) {
  constexpr int NQ = P16 ? 32 : 16;
  const StepDesc* st = p.step;
  const PlanDev* pl = p.plan;
  const int B = st->B, H = p.n_heads;
  volatile int* abort = &sh.abort;
  const uint32_t lanes = static_cast<uint32_t>(warp * 32) << 16;
  const int k = tid;
  TcCursor cur;
  cur.start(sh, B, H, g0);
  tc_write_q<P16>(p, pl->slot_crow[p.slot][cur.b], st->req_nodes[cur.b], cur.h, qbuf, tid);
  fence_async_smem();
  named_bar_sync(kBarSoftmax, 128);
  if (tid == 0) mbar_arrive(&sh.q_full[0]);
  float m[kTcRows], l[kTcRows];
#pragma unroll
  for (int q = 0; q < kTcRows; ++q) {
    m[q] = -INFINITY;
    l[q] = 0.f;
  }
  int seg = 0;
  for (int t = 0; t < n; ++t) {
    const int b = cur.b, kt = cur.kt, nt = cur.nt;
    const bool first = t == 0 || kt == 0;
    const bool last = t == n - 1 || kt == nt - 1;
    const int ctx = st->req_ctx[b], N = st->req_nodes[b], Tk = ctx + N;
    const int key = kt * kTcKeys + k;

    // the next item's q rows are read now, while this tile's scores are being computed, and
    // written into the other Q buffer below
    const bool next_q = first && t + (nt - kt) < n;
    uint4 qraw[2];
    if (next_q) {
      TcCursor nx = cur;
      nx.kt = nx.nt - 1;
      nx.next(sh, B, H);
      tc_load_q(p, pl->slot_crow[p.slot][nx.b], st->req_nodes[nx.b], nx.h, tid, qraw);
    }

    // scores of this key for the block's rows (hi and lo products added)
    bool ok = mbar_wait(&sh.s_full[t & 1], (t >> 1) & 1, abort, p.status);
    if (bar_or<kBarSoftmax>(!ok)) break;
    tc_fence_after();
    float a[NQ];
    tmem_ld_nq<NQ>(tm + lanes + (t & 1) * 32, a);
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(&sh.s_free[t & 1]);
    float s[kTcRows];
#pragma unroll
    for (int q = 0; q < kTcRows; ++q) s[q] = P16 ? a[q] + a[kTcRows + q] : a[q];

    // Q of the next item into the other buffer (the score products of the item before this one,
    // which read it, are complete: their commit preceded this tile's)
    if (next_q) tc_store_q<P16>(qbuf + ((seg + 1) & 1) * kQBytes, tid, qraw);

    // context / ancestor mask (vis bit q: row q sees this key), scale to log2 units
    uint32_t vis = 0;
    if (key < ctx) {
      vis = (1u << N) - 1u;
    } else if (key < Tk) {
      const int j = key - ctx;
      const unsigned long long* anc = st->row_anc + st->req_rowoff[b];
      for (int q = 0; q < N; ++q) vis |= static_cast<uint32_t>((anc[q] >> j) & 1ull) << q;
    }
    bool raise = false;
#pragma unroll
    for (int q = 0; q < kTcRows; ++q) {
      s[q] = ((vis >> q) & 1u) ? s[q] * p.scale_log2 : -INFINITY;
      raise |= s[q] > m[q] + kRaise;
    }

    // P buffer t & 1 is free once PV(t - 2) is complete; in the item's last tile the V rows past
    // its keys (stale cache rows or the next head's) are zeroed so that 0-weights meet finite values
    ok = true;
    if (t >= 2) ok = mbar_wait(&sh.p_free[t & 1], ((t >> 1) - 1) & 1, abort, p.status);
    if (ok && kt == nt - 1) {
      const int s_ = t % kTcStages;
      ok = mbar_wait(&sh.vfull[s_], (t / kTcStages) & 1, abort, p.status);
      if (ok && key >= Tk) {
        uint4* v0 = reinterpret_cast<uint4*>(vring + s_ * kSlotBytes + k * 128);
        uint4* v1 = reinterpret_cast<uint4*>(vring + s_ * kSlotBytes + kBox + k * 128);
#pragma unroll
        for (int i = 0; i < 8; ++i) v0[i] = v1[i] = make_uint4(0, 0, 0, 0);
      }
    }
    if (bar_or<kBarSoftmax>(!ok)) break;

    if (bar_or<kBarSoftmax>(raise)) {
      // new running maxima: the column maxima of the tile over the 128 keys
#pragma unroll
      for (int q = 0; q < kTcRows; ++q) {
        float v = s[q];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
        if (lane == 0) sh.red[warp][q] = v;
      }
      named_bar_sync(kBarSoftmax, 128);
      float alpha[kTcRows];
      bool rescale = false;
#pragma unroll
      for (int q = 0; q < kTcRows; ++q) {
        const float tmax = fmaxf(fmaxf(sh.red[0][q], sh.red[1][q]), fmaxf(sh.red[2][q], sh.red[3][q]));
        const float mn = fmaxf(m[q], tmax);
        alpha[q] = (m[q] == -INFINITY || mn == m[q]) ? 1.f : exp2f(m[q] - mn);
        rescale |= alpha[q] != 1.f;
        m[q] = mn;
      }
      named_bar_sync(kBarSoftmax, 128);  // (sh.red is rewritten by the next raise)
      if (!first && rescale) {
        // O^T *= alpha column by column (both parts) once PV(t - 1) has completed
        ok = mbar_wait(&sh.p_free[(t - 1) & 1], ((t - 1) >> 1) & 1, abort, p.status);
        if (bar_or<kBarSoftmax>(!ok)) break;
        tc_fence_after();
        float o[NQ];
        const uint32_t oaddr = tm + lanes + kOCol + (seg & 1) * 32;
        tmem_ld_nq<NQ>(oaddr, o);
#pragma unroll
        for (int q = 0; q < NQ; ++q) o[q] *= alpha[q & (kTcRows - 1)];
        tmem_st_nq<NQ>(oaddr, o);
        tc_fence_before();
      }
#pragma unroll
      for (int q = 0; q < kTcRows; ++q) l[q] *= alpha[q];
    }

    // weights 2^(s - m) of this key: hi (row q) and lo (row 16 + q) bf16 parts into the P operand
    uint8_t* pb = pbuf + (t & 1) * kPBytes;
#pragma unroll
    for (int q = 0; q < kTcRows; ++q) {
      const float base = m[q] == -INFINITY ? 0.f : m[q];
      const float w = exp2f(s[q] - base);
      l[q] += w;
      const __nv_bfloat16 hi = __float2bfloat16_rn(w);
      *reinterpret_cast<__nv_bfloat16*>(pb + op_off(q, k)) = hi;
      if (P16) *reinterpret_cast<__nv_bfloat16*>(pb + op_off(kTcRows + q, k)) = __float2bfloat16_rn(w - __bfloat162float(hi));
    }
    fence_async_smem();
    named_bar_sync(kBarSoftmax, 128);
    if (tid == 0) {
      mbar_arrive(&sh.p_full[t & 1]);
      if (next_q) mbar_arrive(&sh.q_full[(seg + 1) & 1]);
    }

    if (last) {
      // end of this CTA's part of the item: maxima and per-warp sums to the epilogue (buffer seg & 1,
      // free once the epilogue has taken the part two before)
      ok = seg < 2 || mbar_wait(&sh.h_free[seg & 1], ((seg >> 1) - 1) & 1, abort, p.status);
      if (bar_or<kBarSoftmax>(!ok)) break;
#pragma unroll
      for (int q = 0; q < kTcRows; ++q) {
        float v = l[q];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0) sh.hl[seg & 1][warp][q] = v;
        if (q == k) sh.hm[seg & 1][q] = m[q];
      }
      named_bar_sync(kBarSoftmax, 128);
      if (tid == 0) mbar_arrive(&sh.h_full[seg & 1]);
#pragma unroll
      for (int q = 0; q < kTcRows; ++q) {
        m[q] = -INFINITY;
        l[q] = 0.f;
      }
      ++seg;
    }
    cur.next(sh, B, H);
  }
}

// Epilogue: warps 4-7, thread e owns head-dimension element e (TMEM lane e of O^T).  For each
// item part of the CTA, in order: O (both parts added), the softmax's maxima and sums, then the
// output (whole item), or a partial and -- by the last CTA to finish the item -- the merge of
// all its partials in CTA order.
template <bool P16>
__device__ __forceinline__ void tc_epilogue(const AttnTcParams& p, TcShared& sh, uint32_t tm, int n, long long g0,
                                            long long T, int C, int c, int e, int warp) {
  constexpr int NQ = P16 ? 32 : 16;
  const StepDesc* st = p.step;
  const PlanDev* pl = p.plan;
  const int B = st->B, H = p.n_heads;
  volatile int* abort = &sh.abort;
  const uint32_t lanes = static_cast<uint32_t>((warp & 3) * 32) << 16;
  TcCursor cur;
  cur.start(sh, B, H, g0);
  int t = 0;
  for (int j = 0; t < n; ++j) {
    const int b = cur.b, h = cur.h, nt = cur.nt;
    const int len = min(nt - cur.kt, n - t);  // tiles of this part
    const int N = st->req_nodes[b], crow = pl->slot_crow[p.slot][b];
    bool ok = mbar_wait(&sh.o_full[j & 1], (j >> 1) & 1, abort, p.status);
    ok = ok && mbar_wait(&sh.h_full[j & 1], (j >> 1) & 1, abort, p.status);
    if (bar_or<kBarEpi>(!ok)) break;
    tc_fence_after();
    float a[NQ];
    tmem_ld_nq<NQ>(tm + lanes + kOCol + (j & 1) * 32, a);
    float o[kTcRows], m[kTcRows], L[kTcRows];
#pragma unroll
    for (int q = 0; q < kTcRows; ++q) {
      o[q] = P16 ? a[q] + a[kTcRows + q] : a[q];
      m[q] = sh.hm[j & 1][q];
      L[q] = ((sh.hl[j & 1][0][q] + sh.hl[j & 1][1][q]) + sh.hl[j & 1][2][q]) + sh.hl[j & 1][3][q];
    }
    tc_fence_before();
    named_bar_sync(kBarEpi, 128);
    if (e == 0) {
      mbar_arrive(&sh.o_free[j & 1]);
      mbar_arrive(&sh.h_free[j & 1]);
    }
    const int item = b * H + h;
    const long long gi0 = sh.cum[b] + static_cast<long long>(h) * nt;
    const int cf = tc_cta_of(gi0, T, C), cl = tc_cta_of(gi0 + nt - 1, T, C);
    const int col = h * kTcD + e;
    if (cf == cl) {
#pragma unroll
      for (int q = 0; q < kTcRows; ++q)
        if (q < N) {
          if (!(L[q] > 0.f)) report(p.status, kStatusCheck);
          tc_store_out(p, crow + q, col, L[q] > 0.f ? o[q] / L[q] : 0.f);
        }
    } else {
      const size_t sg = static_cast<size_t>(item + c);
#pragma unroll
      for (int q = 0; q < kTcRows; ++q)
        if (q < N) __stcg(&p.part_o[(sg * kTcRows + q) * kTcD + e], o[q]);
#pragma unroll
      for (int q = 0; q < kTcRows; ++q)
        if (q == e && q < N) {
          __stcg(&p.part_ml[(sg * kTcRows + q) * 2], m[q]);
          __stcg(&p.part_ml[(sg * kTcRows + q) * 2 + 1], L[q]);
        }
      __threadfence();
      named_bar_sync(kBarEpi, 128);
      if (e == 0) {
        int* cnt = p.counters + item;
        const int old = atom_add_acq_rel_gpu(cnt, 1);
        sh.last = old == cl - cf;
        if (sh.last) atomicExch(cnt, 0);
      }
      named_bar_sync(kBarEpi, 128);
      if (sh.last) {
        // online merge of the item's partials in CTA order (one round of loads per partial)
        float M[kTcRows], Ls[kTcRows], O[kTcRows];
#pragma unroll
        for (int q = 0; q < kTcRows; ++q) {
          M[q] = -INFINITY;
          Ls[q] = O[q] = 0.f;
        }
        for (int cc = cf; cc <= cl; ++cc) {
          const size_t s0 = static_cast<size_t>(item + cc) * kTcRows;
          float pm[kTcRows], pl_[kTcRows], po[kTcRows];
#pragma unroll
          for (int q = 0; q < kTcRows; ++q)
            if (q < N) {
              pm[q] = __ldcg(&p.part_ml[(s0 + q) * 2]);
              pl_[q] = __ldcg(&p.part_ml[(s0 + q) * 2 + 1]);
              po[q] = __ldcg(&p.part_o[(s0 + q) * kTcD + e]);
            }
#pragma unroll
          for (int q = 0; q < kTcRows; ++q)
            if (q < N) {
              const float mn = fmaxf(M[q], pm[q]);
              const float mb = mn == -INFINITY ? 0.f : mn;
              const float wa = exp2f(M[q] - mb), wb = exp2f(pm[q] - mb);
              O[q] = O[q] * wa + po[q] * wb;
              Ls[q] = Ls[q] * wa + pl_[q] * wb;
              M[q] = mn;
            }
        }
#pragma unroll
        for (int q = 0; q < kTcRows; ++q)
          if (q < N) {
            if (!(Ls[q] > 0.f)) report(p.status, kStatusCheck);
            tc_store_out(p, crow + q, col, Ls[q] > 0.f ? O[q] / Ls[q] : 0.f);
          }
      }
    }
    t += len;
    if (t < n) {
      cur.kt = cur.nt - 1;
      cur.next(sh, B, H);
    }
  }
}

template <bool P16>
__global__ void __launch_bounds__(kTcThreads, 1) attn_tc_kernel(const AttnTcParams p) {
  constexpr int NQ = P16 ? 32 : 16;
  extern __shared__ uint8_t tc_dyn[];
  __shared__ TcShared sh;
  uint8_t* base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(tc_dyn) + 1023) & ~uintptr_t(1023));
  uint8_t* kring = base;                            // [slot] K box 0, K box 1
  uint8_t* vring = kring + kTcStages * kSlotBytes;  // [slot] V box 0, V box 1
  uint8_t* qbuf = vring + kTcStages * kSlotBytes;   // [2] Q operand
  uint8_t* pbuf = qbuf + 2 * kQBytes;               // [2] P operand
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const StepDesc* st = p.step;
  const PlanDev* pl = p.plan;
  griddep_wait();
  if (p.slot >= pl->n_act) return;
  const int B = st->B, H = p.n_heads;
  if (tid == 0) {
    int acc = 0;
    sh.cum[0] = 0;
    for (int b = 0; b < B; ++b) {
      if (pl->slot_crow[p.slot][b] >= 0) acc += H * ((st->req_ctx[b] + st->req_nodes[b] + kTcKeys - 1) / kTcKeys);
      sh.cum[b + 1] = acc;
    }
    sh.abort = 0;
    for (int i = 0; i < kTcStages; ++i) {
      mbar_init(&sh.kfull[i], 1);
      mbar_init(&sh.kempty[i], 1);
      mbar_init(&sh.vfull[i], 1);
      mbar_init(&sh.vempty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&sh.s_full[i], 1);
      mbar_init(&sh.s_free[i], 4);
      mbar_init(&sh.p_full[i], 1);
      mbar_init(&sh.p_free[i], 1);
      mbar_init(&sh.q_full[i], 1);
      mbar_init(&sh.o_full[i], 1);
      mbar_init(&sh.o_free[i], 1);
      mbar_init(&sh.h_full[i], 1);
      mbar_init(&sh.h_free[i], 1);
    }
    mbar_init(&sh.drain, 1);
    fence_mbar_init();
  }
  __syncthreads();
  // ranges for C = min(grid, T) CTAs, so that every range holds at least one tile (an item's
  // partials then come from every CTA between the ones holding its first and last tiles)
  const long long T = sh.cum[B];
  const int C = static_cast<int>(T < gridDim.x ? T : gridDim.x), c = blockIdx.x;
  if (c >= C) return;  // (the whole CTA)
  const long long g0 = c * T / C, g1 = (c + 1) * T / C;
  const int n = static_cast<int>(g1 - g0);
  if (warp == 0) {
    tmem_alloc(&sh.tmem, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tm = sh.tmem;
  const CUtensorMap* map = p.kv_maps + pl->act_layer[p.slot];
  volatile int* abort = &sh.abort;

  if (warp == 8) {
    // ---------------- TMA producer: K of tile i, then V of tile i - 1 ----------------
    if (lane == 0) {
      prefetch_tmap(map);
      TcCursor ck, cv;
      ck.start(sh, B, H, g0);
      cv = ck;
      const size_t cap = static_cast<size_t>(st->kv_cap);
      auto row_of = [&](const TcCursor& cu, int kv) {
        return static_cast<int>(((static_cast<size_t>(st->req_slot[cu.b]) * 2 + kv) * H + cu.h) * cap) +
               cu.kt * kTcKeys;
      };
      int nk = 0, nv = 0;  // tiles whose K / V copies were issued
      for (int i = 0; i <= n; ++i) {
        if (i < n) {
          const int s = i % kTcStages;
          if (i >= kTcStages && !mbar_wait(&sh.kempty[s], ((i / kTcStages) - 1) & 1, abort, p.status)) break;
          uint8_t* dst = kring + s * kSlotBytes;
          const int row = row_of(ck, 0);
          mbar_arrive_expect_tx(&sh.kfull[s], kSlotBytes);
          tma_load_2d(dst, map, &sh.kfull[s], 0, row);
          tma_load_2d(dst + kBox, map, &sh.kfull[s], 64, row);
          ++nk;
          ck.next(sh, B, H);
        }
        if (i >= 1) {
          const int u = i - 1, s = u % kTcStages;
          if (u >= kTcStages && !mbar_wait(&sh.vempty[s], ((u / kTcStages) - 1) & 1, abort, p.status)) break;
          uint8_t* dst = vring + s * kSlotBytes;
          const int row = row_of(cv, 1);
          mbar_arrive_expect_tx(&sh.vfull[s], kSlotBytes);
          tma_load_2d(dst, map, &sh.vfull[s], 0, row);
          tma_load_2d(dst + kBox, map, &sh.vfull[s], 64, row);
          ++nv;
          cv.next(sh, B, H);
        }
      }
      // the copies issued last into each slot have landed before the kernel returns
      for (int u = nk - 1; u >= 0 && u >= nk - kTcStages; --u) mbar_drain(&sh.kfull[u % kTcStages], (u / kTcStages) & 1);
      for (int u = nv - 1; u >= 0 && u >= nv - kTcStages; --u) mbar_drain(&sh.vfull[u % kTcStages], (u / kTcStages) & 1);
    }
  } else if (warp == 9) {
    // ---------------- MMA issuer: S(t), then PV(t - 1) ----------------
    if (lane == 0) {
      const uint32_t idS = idesc_bf16_m128(NQ), idPV = idesc_bf16_m128(NQ) | (1u << 15);  // (A MN-major)
      const uint32_t k_a = smem_u32(kring), v_a = smem_u32(vring), q_a = smem_u32(qbuf), p_a = smem_u32(pbuf);
      TcCursor cur;
      cur.start(sh, B, H, g0);
      int seg_s = -1, pv_seg = 0;
      bool pv_first = false, pv_last = false;
      // fault injection: CTA 0 issues no MMA, so its softmax's first wait runs out
      const int n_issue = p.withhold && blockIdx.x == 0 ? -1 : n;
      for (int t = 0; t <= n_issue; ++t) {
        bool first = false, last = false;
        if (t < n) {
          first = t == 0 || cur.kt == 0;
          last = t == n - 1 || cur.kt == cur.nt - 1;
          if (first) ++seg_s;
          const int s = t % kTcStages;
          if (!mbar_wait(&sh.kfull[s], (t / kTcStages) & 1, abort, p.status)) break;
          if (t >= 2 && !mbar_wait(&sh.s_free[t & 1], ((t >> 1) - 1) & 1, abort, p.status)) break;
          if (first && !mbar_wait(&sh.q_full[seg_s & 1], (seg_s >> 1) & 1, abort, p.status)) break;
          tc_fence_after();
          const uint32_t kb_a = k_a + s * kSlotBytes, qb_a = q_a + (seg_s & 1) * kQBytes;
          const uint32_t dS = tm + (t & 1) * 32;
#pragma unroll
          for (int kb = 0; kb < 2; ++kb)
#pragma unroll
            for (int k16 = 0; k16 < 4; ++k16)
              umma_bf16(dS, sdesc_sw128(kb_a + kb * kBox + k16 * 32), sdesc_sw128(qb_a + kb * kOpBytes + k16 * 32), idS,
                        (kb | k16) ? 1u : 0u);
          umma_commit(&sh.s_full[t & 1]);
          umma_commit(&sh.kempty[s]);
        }
        if (t >= 1) {
          const int u = t - 1, s = u % kTcStages;
          if (!mbar_wait(&sh.vfull[s], (u / kTcStages) & 1, abort, p.status)) break;
          if (!mbar_wait(&sh.p_full[u & 1], (u >> 1) & 1, abort, p.status)) break;
          if (pv_first && pv_seg >= 2 && !mbar_wait(&sh.o_free[pv_seg & 1], ((pv_seg >> 1) - 1) & 1, abort, p.status))
            break;
          tc_fence_after();
          const uint32_t vb_a = v_a + s * kSlotBytes, pb_a = p_a + (u & 1) * kPBytes;
          const uint32_t dO = tm + kOCol + (pv_seg & 1) * 32;
#pragma unroll
          for (int kk = 0; kk < kTcKeys / 16; ++kk)
            umma_bf16(dO, sdesc_sw128_mn(vb_a + kk * 16 * 128, kBox),
                      sdesc_sw128(pb_a + (kk >> 2) * kOpBytes + (kk & 3) * 32), idPV, (pv_first && kk == 0) ? 0u : 1u);
          umma_commit(&sh.vempty[s]);
          umma_commit(&sh.p_free[u & 1]);
          if (pv_last) umma_commit(&sh.o_full[pv_seg & 1]);
        }
        pv_first = first;
        pv_last = last;
        pv_seg = seg_s;
        if (t < n) cur.next(sh, B, H);
      }
      // every MMA issued has completed before the kernel returns
      umma_commit(&sh.drain);
      mbar_drain(&sh.drain, 0);
    }
  } else if (warp < 4) {
    tc_softmax<P16>(p, sh, tm, qbuf, pbuf, vring, n, g0, tid, warp, lane);
  } else {
    tc_epilogue<P16>(p, sh, tm, n, g0, T, C, c, tid - 128, warp);
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tm, kTmemCols);
  }
}


size_t attn_tc_smem_bytes() { return tc_dyn_smem(); }

size_t attn_tc_partial_rows(int max_batch, int n_heads, int grid) {
  return (static_cast<size_t>(max_batch) * n_heads + grid) * kTcRows;
}

cudaError_t attn_tc_prepare() {
  cudaError_t e = cudaFuncSetAttribute(attn_tc_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(tc_dyn_smem()));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(attn_tc_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(tc_dyn_smem()));
  return e;
}

cudaError_t launch_attention_tc(const AttnTcParams& p, int grid, cudaStream_t s, bool pdl) {
  const dim3 g(grid), blk(kTcThreads);
  return p.o_xs.rows ? launch_k(attn_tc_kernel<true>, g, blk, tc_dyn_smem(), s, pdl, p)
                     : launch_k(attn_tc_kernel<false>, g, blk, tc_dyn_smem(), s, pdl, p);
}

}  // namespace tss
