// Host side of the tensor-core GEMM (mcd_tcgemm.cuh): the SW128 tiling of row-major bf16
// matrices and the stand-alone product behind mcd_tc_gemm (include/mcd_tc.h).
#include <cuda_runtime.h>

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

template <int BN>
__global__ void __launch_bounds__(kThreads, 1) gemm_store_kernel(const GemmArgs g, float* __restrict__ Y) {
  gemm_tile<BN, false, false>(g, [&](int m, int n, float v, float) { Y[(size_t)n * g.M + m] = v; });
}

template <int BN>
static cudaError_t launch_store(const GemmArgs& g, float* Y, cudaStream_t st) {
  cudaError_t e = cudaFuncSetAttribute(gemm_store_kernel<BN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Layout<BN>::kSmemBytes);
  if (e != cudaSuccess) return e;
  gemm_store_kernel<BN><<<dim3(g.N / BN, g.M / kBM), kThreads, Layout<BN>::kSmemBytes, st>>>(g, Y);
  return cudaGetLastError();
}

}  // namespace tc
}  // namespace mcd

using namespace mcd;

extern "C" mcd_status mcd_tc_gemm(int32_t M, int32_t N, int32_t K, int32_t bn, const uint16_t* A, const uint16_t* B,
                                  float* Y, void* stream) {
  if (!A || !B || !Y || M <= 0 || N <= 0 || K <= 0) return MCD_ERR_INVALID_ARG;
  if (M % tc::kBM || K % tc::kBK || (bn != 128 && bn != 256) || N % bn) return MCD_ERR_UNSUPPORTED;
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
    tc::GemmArgs g{ta, nullptr, tb, nullptr, M, N, K, nullptr, err, 2000000000ull};
    e = bn == 256 ? tc::launch_store<256>(g, Y, st) : tc::launch_store<128>(g, Y, st);
  }
  if (e == cudaSuccess) e = cudaMemcpyAsync(&herr, err, sizeof(int), cudaMemcpyDeviceToHost, st);
  if (e == cudaSuccess) e = cudaStreamSynchronize(st);
  cudaFree(ta);
  cudaFree(tb);
  cudaFree(err);
  if (e != cudaSuccess) return cuda_status(e);
  return herr ? (mcd_status)herr : MCD_OK;
}
