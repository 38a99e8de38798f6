// Host side of the tensor-core GEMM (mcd_tcgemm.cuh): the SW128 tiling of row-major bf16
// matrices and the stand-alone product behind mcd_tc_gemm (include/mcd_tc.h).
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>

#include "mcd_host.cuh"
#include "mcd_tcgemm.cuh"
#include "../../include/mcd_tc.h"

namespace mcd {
namespace tc {

// Row-major bf16 [R][K] (row stride ld elements) -> SW128 tiles; one 16-byte chunk per thread.
__global__ void sw128_tile_kernel(const uint16_t* __restrict__ src, int R, int K, int ld, uint8_t* __restrict__ dst) {
  const long long total = (long long)R * (K / 8);
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total; i += (long long)gridDim.x * blockDim.x) {
    const int row = (int)(i / (K / 8)), ch = (int)(i % (K / 8));       // chunk of 8 bf16 along k
    const uint4 v = *reinterpret_cast<const uint4*>(src + (size_t)row * ld + (size_t)ch * 8);
    *reinterpret_cast<uint4*>(dst + sw128_offset(R, row, ch >> 3, ch & 7)) = v;
  }
}

// Stand-alone product: eight warps (two per TMEM lane quarter share the epilogue's columns).
// Launched as a programmatic dependent of the previous kernel in the stream: the grid is set
// up while that kernel runs, and every thread waits for its completion (and the visibility
// of its writes) before the first global access.
constexpr int kStoreThreads = 256;
template <int BN>
__global__ void __launch_bounds__(kStoreThreads, 1) gemm_store_kernel(const GemmArgs g, float* __restrict__ Y) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  asm volatile("griddepcontrol.wait;" ::: "memory");
  gemm_tile<BN, false, false>(g, [&](int m, int n, float v, float) { Y[(size_t)n * g.M + m] = v; });
}

template <int BN>
static cudaError_t launch_store(const GemmArgs& g, float* Y, cudaStream_t st) {
  // the shared-memory opt-in is a property of the function: set once per device
  static std::atomic<unsigned> opted{0};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const unsigned bit = 1u << (dev & 31);
  if (!(opted.load(std::memory_order_acquire) & bit)) {
    e = cudaFuncSetAttribute(gemm_store_kernel<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize, Layout<BN>::kSmemBytes);
    if (e != cudaSuccess) return e;
    opted.fetch_or(bit, std::memory_order_acq_rel);
  }
  const int pitch = g.bn ? g.bn : BN;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((g.N + pitch - 1) / pitch, g.M / kBM);
  cfg.blockDim = dim3(kStoreThreads);
  cfg.dynamicSmemBytes = Layout<BN>::kSmemBytes;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, gemm_store_kernel<BN>, g, Y);
}

// The narrowest instantiation that holds a tile of `pitch` columns (smaller stages: more of
// them in flight).
static cudaError_t launch_store_pitch(const GemmArgs& g, float* Y, cudaStream_t st) {
  const int pitch = g.bn;
  if (pitch <= 128) return launch_store<128>(g, Y, st);
  if (pitch <= 176) return launch_store<176>(g, Y, st);
  return launch_store<256>(g, Y, st);
}

// Tile pitch over N that fills this GPU with one tile per CTA.
static int auto_pitch(int M, int N) {
  int dev = 0, n_sm = 148;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
  return tile_pitch(M, N, n_sm);
}

}  // namespace tc
}  // namespace mcd

using namespace mcd;

extern "C" mcd_status mcd_tc_gemm(int32_t M, int32_t N, int32_t K, int32_t bn, const uint16_t* A, const uint16_t* B,
                                  float* Y, void* stream) {
  if (!A || !B || !Y || M <= 0 || N <= 0 || K <= 0) return MCD_ERR_INVALID_ARG;
  if (M % tc::kBM || K % tc::kBK || (bn != 0 && bn != 128 && bn != 256) || N % (bn ? bn : 16))
    return MCD_ERR_UNSUPPORTED;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t *ta = nullptr, *tb = nullptr;
  int* err = nullptr;
  cudaError_t e = cudaMalloc(&ta, (size_t)M * K * 2);
  if (e == cudaSuccess) e = cudaMalloc(&tb, (size_t)N * K * 2);
  if (e == cudaSuccess) e = cudaMalloc(&err, sizeof(int));
  if (e == cudaSuccess) e = cudaMemsetAsync(err, 0, sizeof(int), st);
  if (e == cudaSuccess) {
    tc::sw128_tile_kernel<<<1024, 256, 0, st>>>(A, M, K, K, ta);
    tc::sw128_tile_kernel<<<1024, 256, 0, st>>>(B, N, K, K, tb);
    e = cudaGetLastError();
  }
  int herr = 0;
  if (e == cudaSuccess) {
    tc::GemmArgs g{ta, nullptr, tb, nullptr, M, N, K, nullptr, err, 2000000000ull, bn ? 0 : tc::auto_pitch(M, N)};
    e = bn == 128 ? tc::launch_store<128>(g, Y, st) : bn == 256 ? tc::launch_store<256>(g, Y, st)
                                                             : tc::launch_store_pitch(g, Y, st);
  }
  if (e == cudaSuccess) e = cudaMemcpyAsync(&herr, err, sizeof(int), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  cudaFree(ta);
  cudaFree(tb);
  cudaFree(err);
  if (e != cudaSuccess) return cuda_status(e);
  return herr ? (mcd_status)herr : MCD_OK;
}

extern "C" mcd_status mcd_tc_tile(int32_t R, int32_t K, int32_t ld, const uint16_t* src, void* dst, void* stream) {
  if (!src || !dst || R <= 0 || K <= 0 || ld < K) return MCD_ERR_INVALID_ARG;
  if (R % 16 || K % tc::kBK || (reinterpret_cast<uintptr_t>(dst) & 1023u) || (reinterpret_cast<uintptr_t>(src) & 15u) ||
      ld % 8)
    return MCD_ERR_UNSUPPORTED;
  tc::sw128_tile_kernel<<<1024, 256, 0, static_cast<cudaStream_t>(stream)>>>(src, R, K, ld,
                                                                             static_cast<uint8_t*>(dst));
  return cuda_status(cudaGetLastError());
}

extern "C" mcd_status mcd_tc_gemm_tiled(int32_t M, int32_t N, int32_t K, int32_t bn, const void* A_tiled,
                                        const void* B_tiled, float* Y, int32_t* err, void* stream) {
  if (!A_tiled || !B_tiled || !Y || !err || M <= 0 || N <= 0 || K <= 0) return MCD_ERR_INVALID_ARG;
  if (M % tc::kBM || K % tc::kBK || (bn != 0 && bn != 128 && bn != 256) || N % (bn ? bn : 16))
    return MCD_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(A_tiled) | reinterpret_cast<uintptr_t>(B_tiled)) & 1023u) return MCD_ERR_UNSUPPORTED;
  tc::GemmArgs g{static_cast<const uint8_t*>(A_tiled), nullptr, static_cast<const uint8_t*>(B_tiled), nullptr,
                 M, N, K, nullptr, err, 2000000000ull, bn ? 0 : tc::auto_pitch(M, N)};
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  return cuda_status(bn == 128   ? tc::launch_store<128>(g, Y, st)
                     : bn == 256 ? tc::launch_store<256>(g, Y, st)
                                 : tc::launch_store_pitch(g, Y, st));
}
