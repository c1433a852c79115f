// tss_linear_static: the weight-streaming linear layer without any device allocation.
//
// Some callers cannot allocate device memory when they need this layer: a plugin living inside a
// host framework that owns the whole device memory pool, a process whose memory budget is fixed
// at start-up, or a latency-critical loop that must not call cudaMalloc/cudaFree because those
// calls can synchronise the whole device and stall unrelated streams.  tss_linear needs a
// tss_ctx, and tss_create allocates the stream-K scratch (partial tiles and per-tile counters).
// This entry point runs the same GEMM kernel with that scratch taken from file-scope device
// arrays instead, so it needs no context and allocates nothing.
//
// The arrays belong to this file's CUDA module, which the runtime loads on a device (lazily, at
// the first call on that device, under CUDA's default lazy module loading): from then on the GPU
// holds them (kStaticPartialBytes + counters + a status word) until the process exits.  A caller
// that hands the rest of the device memory to its own pool should make one call first.  Every
// call on a device shares them, so two calls that overlap on the GPU (different streams, or
// different host threads) race and may return wrong results; serialise them on one stream.
#include <cudaTypedefs.h>

#include <mutex>
#include <string>

#include "internal.h"

namespace {

constexpr size_t kStaticPartialBytes = size_t(8) << 20;  // 8 MiB of stream-K partial tiles
constexpr size_t kStaticPartialFloats = kStaticPartialBytes / sizeof(float);
constexpr int kStaticCounters = 256;                      // per-tile counters: n_out <= 256 * 128
constexpr int kStaticMaxRows = 64;
constexpr int kMaxDevices = 64;

static __device__ __align__(256) float g_static_partials[kStaticPartialFloats];
static __device__ __align__(256) int g_static_counters[kStaticCounters];
// First failure of a device-side check or bounded wait since the last tss_linear_static_status
// (0: none); the GEMM kernel records it and never traps.
static __device__ __align__(256) int g_static_status;

struct DeviceScratch {
  bool ready = false;
  float* partials = nullptr;  // device addresses of the arrays above on this device
  int* counters = nullptr;
  int* status = nullptr;
  int num_sms = 0;
};
DeviceScratch g_dev[kMaxDevices];
std::mutex g_mu;
std::once_flag g_encode_once;
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

bool encode(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint32_t box_rows, int rank) {
  std::call_once(g_encode_once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  const PFN_cuTensorMapEncodeTiled_v12000 fn = g_encode;
  if (!fn) return false;
  cuuint64_t dims[3] = {inner, rows, 1};
  cuuint64_t strides[2] = {inner * 2, inner * rows * 2};
  cuuint32_t box[3] = {64, box_rows, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, static_cast<cuuint32_t>(rank), const_cast<void*>(base), dims, strides,
            box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

tss_status reject(tss_status s, const std::string& msg) {
  tss::set_last_error(msg);
  return s;
}

// Once per device, with that device current: find the arrays' device addresses (in host code
// their names are only host-side stand-ins) and set the kernel's shared-memory limit.
tss_status setup_device(int dev, DeviceScratch** out) {
  std::lock_guard<std::mutex> lock(g_mu);
  DeviceScratch& d = g_dev[dev];
  if (!d.ready) {
    int major = 0, minor = 0;
    cudaError_t e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    if (e != cudaSuccess) return reject(TSS_ERR_CUDA, std::string("cudaDeviceGetAttribute: ") + cudaGetErrorString(e));
    if (major != 10 || minor != 3) return reject(TSS_ERR_UNSUPPORTED_ARCH, "tss_linear_static needs an sm_103 GPU");
    e = cudaDeviceGetAttribute(&d.num_sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return reject(TSS_ERR_CUDA, std::string("cudaDeviceGetAttribute: ") + cudaGetErrorString(e));
    e = cudaGetSymbolAddress(reinterpret_cast<void**>(&d.partials), g_static_partials);
    if (e != cudaSuccess) return reject(TSS_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
    e = cudaGetSymbolAddress(reinterpret_cast<void**>(&d.counters), g_static_counters);
    if (e != cudaSuccess) return reject(TSS_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
    e = cudaGetSymbolAddress(reinterpret_cast<void**>(&d.status), g_static_status);
    if (e != cudaSuccess) return reject(TSS_ERR_CUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
    e = tss::gemm_prepare(232448);  // the per-block shared-memory maximum of sm_103 (227 KiB)
    if (e != cudaSuccess) return reject(TSS_ERR_CUDA, std::string("cudaFuncSetAttribute: ") + cudaGetErrorString(e));
    d.ready = true;
  }
  *out = &d;
  return TSS_OK;
}

}  // namespace

extern "C" tss_status tss_linear_static(const void* x, const void* w, float* y, int m_rows, int k_dim, int n_out,
                                        void* stream) {
  if (!x || !w || !y) return reject(TSS_ERR_INVALID_ARG, "NULL argument");
  if (m_rows < 1 || m_rows > kStaticMaxRows) return reject(TSS_ERR_INVALID_ARG, "m_rows must be in [1, 64]");
  if (k_dim < 64 || k_dim % 64 != 0) return reject(TSS_ERR_INVALID_ARG, "k_dim must be a positive multiple of 64");
  if (n_out < 128 || n_out % 128 != 0 || n_out / 128 > kStaticCounters)
    return reject(TSS_ERR_INVALID_ARG, "n_out must be a multiple of 128 in [128, 32768]");
  if ((reinterpret_cast<uintptr_t>(x) & 15u) || (reinterpret_cast<uintptr_t>(w) & 15u))
    return reject(TSS_ERR_INVALID_ARG, "x and w must be 16-byte aligned");
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return reject(TSS_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return reject(TSS_ERR_UNSUPPORTED_ARCH, "device index beyond 63");
  DeviceScratch* ds = nullptr;
  tss_status st = setup_device(dev, &ds);
  if (st != TSS_OK) return st;

  const int n_pad = (m_rows + 15) / 16 * 16;
  const int n_tiles = n_out / 128, kb = k_dim / 64;
  const long long T = static_cast<long long>(n_tiles) * kb;
  const int grid = static_cast<int>(T < ds->num_sms ? T : ds->num_sms);  // one CTA per SM
  const size_t need = static_cast<size_t>(grid + n_tiles) * 128 * n_pad;
  if (need > kStaticPartialFloats)
    return reject(TSS_ERR_INVALID_ARG, "problem needs " + std::to_string(need * 4) +
                                           " bytes of stream-K scratch; the static limit is 8 MiB");
  int stages = 2;
  while (stages < 12 && tss::gemm_smem_bytes(n_pad, stages + 1) <= 220 * 1024) ++stages;
  CUtensorMap tx, tw;
  if (!encode(&tx, x, k_dim, m_rows, n_pad, 2) || !encode(&tw, w, k_dim, n_out, 128, 3))
    return reject(TSS_ERR_CUDA, "cuTensorMapEncodeTiled failed");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // The counters must start at zero; a call cut short by a device timeout could leave them set.
  e = cudaMemsetAsync(ds->counters, 0, sizeof(int) * n_tiles, s);
  if (e != cudaSuccess) return reject(TSS_ERR_CUDA, std::string("cudaMemsetAsync: ") + cudaGetErrorString(e));
  tss::GemmParams g{};
  g.n_tiles = n_tiles;
  g.kb = kb;
  g.n_pad = n_pad;
  g.stages = stages;
  g.n_acc_bufs = 2;
  g.slot = -1;
  g.m_raw = m_rows;
  g.layer_fixed = 0;
  g.partials = ds->partials;
  g.counters = ds->counters;
  g.status = ds->status;
  g.out = y;
  g.out_ld = n_out;
  g.o_real = n_out;
  e = tss::launch_gemm(tss::kEpiStore, tw, tx, g, grid, tss::gemm_smem_bytes(n_pad, stages), s, false);
  if (e != cudaSuccess) return reject(TSS_ERR_CUDA, std::string("launch: ") + cudaGetErrorString(e));
  return TSS_OK;
}

// Synchronise `stream`, then return and clear the status word of the current device.
extern "C" tss_status tss_linear_static_status(void* stream) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return reject(TSS_ERR_CUDA, std::string("cudaGetDevice: ") + cudaGetErrorString(e));
  if (dev < 0 || dev >= kMaxDevices) return reject(TSS_ERR_UNSUPPORTED_ARCH, "device index beyond 63");
  DeviceScratch* ds = nullptr;
  tss_status st = setup_device(dev, &ds);
  if (st != TSS_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int v = 0;
  e = cudaStreamSynchronize(s);
  if (e == cudaSuccess) e = cudaMemcpy(&v, ds->status, sizeof(int), cudaMemcpyDeviceToHost);
  if (e == cudaSuccess) e = cudaMemset(ds->status, 0, sizeof(int));
  if (e != cudaSuccess) return reject(TSS_ERR_CUDA, std::string("status read: ") + cudaGetErrorString(e));
  if (v != 0) return reject(v, std::string("device status of tss_linear_static: ") + tss_status_string(v));
  return TSS_OK;
}
