// Split-KV attention of a draft block over its request's KV cache, with the chain/tree mask.
//
// For request b, head h and draft-block row i (App. "Models": rotary multi-head attention of a
// LLaMA block; the draft block is scored in parallel, Sec. "Problem Formulation"):
//   o_i = softmax_j(q_i . k_j / sqrt(D)) v_j over every context key j < ctx_len and every block
//   key ctx_len + t for which block row t is row i itself or one of its ancestors.
// The block's own K/V rows were appended to the cache by the QKV epilogue, so all keys are read
// from the cache.  The key range [0, ctx_len + N) is cut into 64-key tiles and the tiles into
// splits; each CTA (split, head, request) runs an online softmax over its tiles with bf16
// mma.sync (queries = M side, 16 rows per warp), writes an unnormalised partial (O, max, sum),
// and the last CTA of (request, head) to finish merges the partials in split order.
//
// Only requests that run this layer are visited (the controller's per-slot list); a request that
// skips the layer reads none of its KV.  Blocks of more than 64 rows take the wide variant: 256
// threads, eight 16-row query tiles (one warp each), buffers for 128 rows.
#include "attn_body.cuh"

namespace tss {

size_t attn_smem_bytes(int head_dim) { return attn_smem_bytes_impl(head_dim); }

template <int D, bool P16, bool WIDE>
__global__ void __launch_bounds__(WIDE ? 2 * kAttnThreads : kAttnThreads) attn_kernel(const AttnParams p) {
  constexpr int NT = WIDE ? 2 * kAttnThreads : kAttnThreads;
  extern __shared__ __align__(16) uint8_t smem_raw[];
  __shared__ float sM[NT / 32][16], sL[NT / 32][16];
  __shared__ int s_last;
  griddep_wait();
  griddep_launch();
  attention_item<D, 0, P16, WIDE ? kMaxNodes : kNarrowNodes, NT>(p, blockIdx.x, blockIdx.y, blockIdx.z, threadIdx.x,
                                                                 smem_raw, sM, sL, &s_last);
}

template <int D, bool P16, bool WIDE>
static size_t attn_kernel_smem() {
  return WIDE ? attn_wide_smem_bytes(D) : attn_smem_bytes(D) + (P16 ? attn_qlo_bytes(D) : 0);
}

template <int D, bool P16, bool WIDE>
static cudaError_t attn_prepare_one() {
  cudaError_t e = cudaFuncSetAttribute(attn_kernel<D, P16, WIDE>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                       cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(attn_kernel<D, P16, WIDE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(attn_kernel_smem<D, P16, WIDE>()));
}

cudaError_t attn_prepare() {
  cudaError_t e = attn_prepare_one<64, false, false>();
  if (e == cudaSuccess) e = attn_prepare_one<128, false, false>();
  if (e == cudaSuccess) e = attn_prepare_one<64, true, false>();
  if (e == cudaSuccess) e = attn_prepare_one<128, true, false>();
  if (e == cudaSuccess) e = attn_prepare_one<64, false, true>();
  if (e == cudaSuccess) e = attn_prepare_one<128, false, true>();
  if (e == cudaSuccess) e = attn_prepare_one<64, true, true>();
  if (e == cudaSuccess) e = attn_prepare_one<128, true, true>();
  return e;
}

template <int D>
static cudaError_t launch_d(const AttnParams& p, dim3 grid, cudaStream_t s, bool pdl) {
  const bool p16 = p.o_xs.rows != 0;  // the persistent path's operands and precision
  const dim3 narrow(kAttnThreads), wide(2 * kAttnThreads);
  if (p.wide)
    return p16 ? launch_k(attn_kernel<D, true, true>, grid, wide, attn_kernel_smem<D, true, true>(), s, pdl, p)
               : launch_k(attn_kernel<D, false, true>, grid, wide, attn_kernel_smem<D, false, true>(), s, pdl, p);
  return p16 ? launch_k(attn_kernel<D, true, false>, grid, narrow, attn_kernel_smem<D, true, false>(), s, pdl, p)
             : launch_k(attn_kernel<D, false, false>, grid, narrow, attn_kernel_smem<D, false, false>(), s, pdl, p);
}

cudaError_t launch_attention(const AttnParams& p, int B, cudaStream_t s, bool pdl) {
  const dim3 grid(p.n_splits, p.n_heads, B);
  if (p.head_dim == 64) return launch_d<64>(p, grid, s, pdl);
  if (p.head_dim == 128) return launch_d<128>(p, grid, s, pdl);
  return cudaErrorInvalidValue;
}

}  // namespace tss
