// Split-K tensor-core GEMM that allocates nothing: its partial sums and its error
// word live in file-scope static device arrays instead of memory from cudaMalloc.
//
// Some callers cannot allocate device memory when they call us: a host framework
// that owns every device allocation through its own pool, or a latency-critical
// loop in which a cudaMalloc would synchronise the device.  This entry point lets
// them run the bf16 GEMM C = A B^T split over K with no allocation at all.
//
// The K range is cut into `splits` slices of whole 64-wide blocks; slice s runs the
// library's tensor-core GEMM kernel on A[:, Ks] and B[:, Ks] into scratch slice s,
// then a reduction kernel adds the slices in order into C.
#include <cudaTypedefs.h>

#include <mutex>

#include "../../include/hero.h"
#include "hero_internal.cuh"

namespace hero {
namespace {

// Shared by every call on a device; holds the last call's contents until exit.
constexpr size_t kNoAllocScratchFloats = (size_t)4 << 20;   // 16 MiB of fp32 partial sums
__device__ __align__(256) float g_noalloc_scratch[kNoAllocScratchFloats];
__device__ __align__(256) uint32_t g_noalloc_err[64];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mu;
float* g_scratch_ptr[kMaxDevices] = {};
uint32_t* g_err_ptr[kMaxDevices] = {};

PFN_cuTensorMapEncodeTiled_v12000 g_enc = nullptr;

bool encode(CUtensorMap* tm, const void* ptr, uint64_t inner, uint64_t outer, uint64_t row_bytes,
            uint32_t box_outer) {
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {64, box_outer};
  cuuint32_t es[2] = {1, 1};
  return g_enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box,
               es, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

__global__ void k_splitk_reduce(const float* __restrict__ part, float* __restrict__ C, long mn,
                                int splits) {
  for (long i = (long)blockIdx.x * blockDim.x + threadIdx.x; i < mn; i += (long)gridDim.x * blockDim.x) {
    float s = 0.f;
    for (int k = 0; k < splits; ++k) s += part[(size_t)k * mn + i];  // fixed order
    C[i] = s;
  }
}

hero_status fail_na(hero_status s, const char* m) {
  set_last_error(m);
  return s;
}

}  // namespace
}  // namespace hero

using namespace hero;

extern "C" hero_status hero_gemm_bf16_splitk_noalloc(const uint16_t* A, const uint16_t* B, float* C,
                                                     int32_t M, int32_t N, int32_t K,
                                                     int32_t splits, void* cuda_stream) {
  set_last_error("");
  if (!A || !B || !C || M < 1 || N < 8 || N % 8 != 0 || K < 64 || K % 64 != 0 || splits < 1)
    return fail_na(HERO_ERR_ARG,
                   "need non-NULL pointers, M >= 1, N a multiple of 8, K a multiple of 64, splits >= 1");
  const int kblocks = K / 64;
  if (splits > kblocks) return fail_na(HERO_ERR_ARG, "splits exceeds K / 64");
  if ((size_t)splits * (size_t)M * (size_t)N > kNoAllocScratchFloats)
    return fail_na(HERO_ERR_ARG,
                   "splits * M * N exceeds the static scratch of 4194304 fp32 partial sums");
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return fail_na(HERO_ERR_CUDA, "no usable current device");
  {
    // One-time set-up per device (with that device current): resolve the
    // device addresses of the static arrays; host code must not pass the
    // symbols themselves to a kernel.
    std::lock_guard<std::mutex> lk(g_setup_mu);
    if (!g_enc) {
      void* fn = nullptr;
      cudaDriverEntryPointQueryResult q;
      if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                           &q) != cudaSuccess ||
          q != cudaDriverEntryPointSuccess)
        return fail_na(HERO_ERR_CUDA, "cuTensorMapEncodeTiled is not available from the driver");
      g_enc = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    if (!g_scratch_ptr[dev]) {
      void* p = nullptr;
      void* e = nullptr;
      if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess ||
          cudaGetSymbolAddress(&e, g_noalloc_err) != cudaSuccess)
        return fail_na(HERO_ERR_CUDA, "cudaGetSymbolAddress failed for the static scratch");
      g_scratch_ptr[dev] = static_cast<float*>(p);
      g_err_ptr[dev] = static_cast<uint32_t*>(e);
    }
  }
  int sms = 0;
  if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return fail_na(HERO_ERR_CUDA, "cudaDeviceGetAttribute failed");
  cudaStream_t st = static_cast<cudaStream_t>(cuda_stream);
  float* scratch = g_scratch_ptr[dev];
  uint32_t* err = g_err_ptr[dev];
  // A sticky error from earlier work on this thread would otherwise be taken for a
  // failure of the reduction launch below; report it without enqueueing anything.
  if (cudaPeekAtLastError() != cudaSuccess)
    return fail_na(HERO_ERR_CUDA, "a CUDA error from earlier work is pending on this thread");
  // The error word of the previous call is not cleared here: the status query reports
  // (and clears) it.  The GEMM only ever sets bits, so one query after a sequence of
  // calls reports a failure of any of them.
  for (int s = 0; s < splits; ++s) {
    // slice s owns K blocks [s kblocks / splits, (s + 1) kblocks / splits): never
    // empty, since splits <= kblocks
    const int kb0 = (int)((long)s * kblocks / splits);
    const int kb1 = (int)((long)(s + 1) * kblocks / splits);
    const uint64_t kk = (uint64_t)(kb1 - kb0) * 64;
    CUtensorMap ta, tb;
    if (!encode(&ta, A + (size_t)kb0 * 64, kk, M, (uint64_t)K * 2, 128) ||
        !encode(&tb, B + (size_t)kb0 * 64, kk, N, (uint64_t)K * 2, 256))
      return fail_na(HERO_ERR_CUDA, "tensor map encoding failed");
    GemmArgs g{};
    g.m_static = M;
    g.m_max = M;
    g.N = N;
    g.K = (int)kk;
    g.out_f32 = scratch + (size_t)s * M * N;
    g.ldo = N;
    g.err = err;
    if (launch_gemm_tc(256, EPI_STORE_F32, ta, tb, g, sms, st) != cudaSuccess)
      return fail_na(HERO_ERR_CUDA, "GEMM launch failed");
  }
  const long mn = (long)M * N;
  long blocks = (mn + 255) / 256;
  if (blocks > 4096) blocks = 4096;
  cudaLaunchConfig_t lc = {};
  lc.gridDim = dim3((unsigned)blocks);
  lc.blockDim = dim3(256);
  lc.stream = st;
  if (cudaLaunchKernelEx(&lc, k_splitk_reduce, (const float*)scratch, C, mn, (int)splits) !=
      cudaSuccess)
    return fail_na(HERO_ERR_CUDA, "reduction launch failed");
  return HERO_OK;
}

extern "C" hero_status hero_gemm_bf16_splitk_noalloc_status(void* cuda_stream) {
  set_last_error("");
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
    return fail_na(HERO_ERR_CUDA, "no usable current device");
  uint32_t* err = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_setup_mu);
    err = g_err_ptr[dev];
  }
  if (!err) return HERO_OK;   // no call has run on this device
  if (cudaStreamSynchronize(static_cast<cudaStream_t>(cuda_stream)) != cudaSuccess)
    return fail_na(HERO_ERR_CUDA, "stream synchronisation failed");
  uint32_t e = 0;
  if (cudaMemcpy(&e, err, sizeof(e), cudaMemcpyDeviceToHost) != cudaSuccess)
    return fail_na(HERO_ERR_CUDA, "reading the static error word failed");
  if (e && cudaMemset(err, 0, sizeof(e)) != cudaSuccess)
    return fail_na(HERO_ERR_CUDA, "clearing the static error word failed");
  return status_of_error_word(e);
}
