// Shared device-side definitions of the TSS verification library (sm_103a).
//
// Layout of the per-step descriptor the host uploads, of the controller's plan, and inline-PTX
// wrappers for the Blackwell primitives the kernels use: mbarrier, TMA (cp.async.bulk.tensor),
// tcgen05 (TMEM alloc, UMMA, commit, TMEM loads), programmatic dependent launch, and the
// legacy warp-level mma.sync/ldmatrix used by the attention kernel.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/tss.h"

namespace tss {

constexpr int kMaxLayers = 64;
constexpr int kMaxBatch = 64;
constexpr int kMaxRows = 256;
constexpr int kMaxNodes = 128;    // rows of one request's draft block (root included)
constexpr int kNarrowNodes = 64;  // blocks the attention inside the persistent kernel takes (larger: the
                                  // separate attention kernel's wide variant)
constexpr int kMaxSplits = 16;  // key splits of one (request, head) in the attention
constexpr int kFinalSlot = kMaxLayers;  // plan slot of the final norm + LM head (all rows)
constexpr int kPathStride = kMaxNodes;  // internal copy of each request's accepted path

// Device status word codes (mirrors tss_status).
constexpr int kStatusOk = 0;
constexpr int kStatusTimeout = TSS_ERR_TIMEOUT;
constexpr int kStatusCheck = TSS_ERR_DEVICE_CHECK;

// Per-verify descriptor, written by the host into pinned memory and copied to the device before
// the step's kernels run.  Fixed size so that a captured CUDA graph reads it from one address.
struct StepDesc {
  int B, M, n_act_host, mode;
  float inv_temperature;
  int uniform_stride, path_stride, kv_cap;
  uint32_t seed_lo, seed_hi, off_lo, off_hi;
  int req_ctx[kMaxBatch];
  int req_nodes[kMaxBatch];
  int req_rowoff[kMaxBatch];
  int req_slot[kMaxBatch];
  int req_domain[kMaxBatch];
  // S(x) of every request: the domain map's entry for its domain when the step was enqueued (the
  // lookup S(x) = Phi(d(x)) runs on the host, so a later change of the map affects later steps
  // only), 0 (dense) for a domain that is not configured.
  unsigned long long req_phi[kMaxBatch];
  int req_rng[kMaxBatch];  // request index of the Philox counter (the caller's index when a batch is split)
  int row_req[kMaxRows];
  int row_pos[kMaxRows];
  int row_parent[kMaxRows];  // request-local parent, -1 for the root
  unsigned long long row_anc[kMaxRows];     // request-local ancestor-or-self bits of block rows 0..63
  unsigned long long row_anc_hi[kMaxRows];  // ... and of block rows 64..127
  const int* tokens;
  const float* draft_probs;
  const float* uniforms;
  int* accept_len;
  int* bonus;
  int* path;
  int* new_ctx;
  float* logits;
  __nv_bfloat16* kv_layer[kMaxLayers];
};

// Written on the device by the skip controller from the descriptor and the domain table Phi.
struct PlanDev {
  int n_act;                      // layers in the union of the batch's active sets
  int act_layer[kMaxLayers + 1];  // slot -> layer, ascending
  unsigned long long req_mask[kMaxBatch];     // S(x) of every request
  int slot_M[kMaxLayers + 1];                 // rows that run slot j (slot kFinalSlot: all)
  int slot_rows[kMaxLayers + 1][kMaxRows];    // compacted row list of slot j
  int slot_crow[kMaxLayers + 1][kMaxBatch];   // first compacted row of request b, -1 if skipped
  int res_accept[kMaxBatch];                  // acceptance results kept for the compaction kernel
  int res_path[kMaxBatch][kPathStride];
};

// ------------------------------------------------------------------------------------------
// Status reporting: record the first failure; never trap.
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ void report(int* status, int code) {
  if (status) atomicCAS(status, 0, code);
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s bound on every spin

// Arrival on a cross-CTA counter with release and acquire semantics at GPU scope.  Issued by one
// thread after a CTA barrier, its release covers the stores every thread of the CTA made before
// that barrier, and its acquire (with a barrier after it) orders the CTA's later loads after
// the other arrivals' stores: the fences around the counter are in the atomic itself.
__device__ __forceinline__ int atom_add_acq_rel_gpu(int* p, int v) {
  int old;
  asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}

// ------------------------------------------------------------------------------------------
// Programmatic dependent launch
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch() { asm volatile("griddepcontrol.launch_dependents;"); }

// ------------------------------------------------------------------------------------------
// Shared-memory addresses, mbarriers
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// Same, but the thread may stay suspended in the instruction for up to `hint_ns` nanoseconds
// while the phase is incomplete (it resumes when the phase completes): a waiting thread then
// takes no issue slots from the other warps of its SM sub-partition.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t* bar, uint32_t parity, uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait for the phase with the given parity.  On expiry (or if *abort is already set) it
// raises *abort, records TIMEOUT and returns false.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity, volatile int* abort, int* status) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 255) == 0) {
      if (*abort) return false;
      if (globaltimer_ns() - t0 > kWaitLimitNs) {
        *abort = 1;
        report(status, kStatusTimeout);
        return false;
      }
    }
  }
}

// ------------------------------------------------------------------------------------------
// TMA tiled loads (global -> shared, completion on an mbarrier)
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ void prefetch_tmap(const CUtensorMap* m) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(m)) : "memory");
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* m, uint64_t* bar, int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4}], [%2];" ::"r"(
          smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(smem_u32(bar)), "r"(c0), "r"(c1)
      : "memory");
}

__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* m, uint64_t* bar, int c0, int c1, int c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(
          smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(m)), "r"(smem_u32(bar)), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}

// Linear bulk copy global -> shared of `bytes` (multiple of 16, both addresses 16-byte aligned).
// L2 policy for data read exactly once (streamed weights): evicted before anything else.
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
__device__ __forceinline__ void bulk_load_hint(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                               uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}
__device__ __forceinline__ void bulk_load(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                   smem_u32(dst)),
               "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void bulk_prefetch_l2(const void* src, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(reinterpret_cast<uint64_t>(src)), "r"(bytes)
               : "memory");
}

// Weights are stored pre-tiled: for each 128-row x 64-column block (16 KiB) the exact byte image
// that a 128-byte-swizzled TMA box of it would leave in shared memory, blocks ordered
// [layer][row tile][k-block].  One linear bulk copy then fills a pipeline stage.
constexpr uint32_t kTileBytes = 128 * 64 * 2;
constexpr size_t kTileElems = 128 * 64;

// Activation (B) operands of the persistent kernel use the same idea: per 64-column k-block,
// contiguous [rows][64] bf16 blocks in 128-byte-swizzled order, so the operand of consecutive
// k-blocks is one linear bulk copy.  Each activation x is kept as two bf16 parts, hi = bf16(x)
// and lo = bf16(x - hi); the GEMM multiplies both by the weights, so the activation keeps about
// 16 significant bits while the tensor cores see bf16 only.  For up to 128 token rows M both
// parts share one block: hi in row j, lo in row half + j (half = xs_half(M)), one MMA of width
// rows = pad16(half + M) yields W.hi and W.lo in separate accumulator columns, and the epilogue
// adds them in fp32.  Beyond that (parts = 2) hi and lo are consecutive blocks of pad16(M) rows
// and two MMAs accumulate into the same columns.
struct XsLayout {
  int rows;   // rows of one block (the MMA width N); 0: plain row-major [row][K] bf16
  int parts;  // 1: hi and lo in one block; 2: a hi block then a lo block per k-block
  int half;   // parts == 1: row offset of the lo part
};
__host__ __device__ inline int xs_half(int M) { return M <= 8 ? 8 : (M + 15) & ~15; }
__host__ __device__ inline XsLayout xs_layout(int M) {
  const int half = xs_half(M);
  if (half + M <= 256) return XsLayout{(half + M + 15) & ~15, 1, half};
  return XsLayout{(M + 15) & ~15, 2, 0};
}
// (32-bit index arithmetic: an operand holds at most 2 x 256 rows x 32768 columns)
__host__ __device__ __forceinline__ uint32_t xs_elem(const XsLayout& L, int j, int k, int lo) {
  const uint32_t kb = static_cast<uint32_t>(k) >> 6, kc = static_cast<uint32_t>(k) & 63u;
  const uint32_t part = L.parts == 2 ? static_cast<uint32_t>(lo) : 0u;
  const uint32_t row = static_cast<uint32_t>(L.parts == 1 && lo ? L.half + j : j);
  return ((kb * L.parts + part) * L.rows + row) * 64u + ((((kc >> 3) ^ (row & 7u)) << 3) | (kc & 7u));
}
__device__ __forceinline__ void store_split(__nv_bfloat16* buf, const XsLayout& L, int j, int k, float x) {
  const __nv_bfloat16 hi = __float2bfloat16_rn(x);
  buf[xs_elem(L, j, k, 0)] = hi;
  buf[xs_elem(L, j, k, 1)] = __float2bfloat16_rn(x - __bfloat162float(hi));
}

// ------------------------------------------------------------------------------------------
// tcgen05: tensor memory and the 5th-generation MMA
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ void tmem_alloc(uint32_t* dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// Shared-memory matrix descriptor for a K-major operand stored with the 128-byte swizzle that a
// TMA box of 64 bf16 (128 B) x rows produces: rows of 128 B, 8-row groups 1024 B apart.
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);  // start address >> 4
  d |= static_cast<uint64_t>(1) << 16;                   // leading byte offset (unused for SW128 K-major)
  d |= static_cast<uint64_t>(1024 >> 4) << 32;           // stride byte offset: 8 rows * 128 B
  d |= static_cast<uint64_t>(1) << 46;                   // descriptor version for tcgen05
  d |= static_cast<uint64_t>(2) << 61;                   // swizzle mode: 128 B
  return d;
}

// Instruction descriptor, kind::f16: bf16 A and B (K-major), fp32 accumulator, M = 128.
__host__ __device__ constexpr uint32_t idesc_bf16_m128(int n) {
  return (1u << 4)                               // D format: f32
         | (1u << 7)                             // A format: bf16
         | (1u << 10)                            // B format: bf16
         | (static_cast<uint32_t>(n >> 3) << 17)  // N >> 3
         | (static_cast<uint32_t>(128 >> 4) << 24);  // M >> 4
}

__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

// 32 lanes x 16 columns of 32-bit TMEM cells -> 16 registers per thread (thread i reads lane i).
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float* v) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, "
      "[%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]), "=r"(r[8]),
        "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// ------------------------------------------------------------------------------------------
// Warp-level tensor-core MMA (attention) and ldmatrix
// ------------------------------------------------------------------------------------------
__device__ __forceinline__ void mma_bf16_16816(float* d, const uint32_t* a, const uint32_t* b) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

__device__ __forceinline__ void mma_f16_16816(float* d, const uint32_t* a, const uint32_t* b) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

__device__ __forceinline__ uint32_t pack_f16(float lo, float hi) {
  __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Two bf16 values (low half first) to two fp16 values, round to nearest.
__device__ __forceinline__ uint32_t bf16x2_to_f16x2(uint32_t v) {
  const float lo = __uint_as_float(v << 16), hi = __uint_as_float(v & 0xffff0000u);
  uint32_t r;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
  return r;
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t* r, const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}

__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t* r, const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void named_bar_sync(int id, int nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}

}  // namespace tss
