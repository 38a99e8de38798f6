// mcd_topk_softmax_static: the top-k / temperature distributions of mcd_topk_softmax for
// callers that must not allocate device memory.  Its per-row records live in one
// file-scope __device__ array (kStaticTopkRows records) instead of context scratch, so
// the call needs no mcd_ctx (whose creation allocates) and allocates nothing itself.
#include <atomic>
#include <cmath>
#include <mutex>

#include "mcd_internal.cuh"
#include "mcd_sampler.cuh"

namespace mcd {
namespace {

constexpr int kStaticTopkRows = MCD_STATIC_TOPK_MAX_ROWS;
constexpr int kMaxDevices = 64;

// Scratch records, one per logits row.  Nothing here needs to start at zero: block_topk
// writes every field a row's copy-out reads before it is read.
__device__ __align__(256) TopkRec g_topk_scratch[kStaticTopkRows];

// Per-device address of the scratch.  After the first call on a device every call reads it
// with one acquire load and takes no lock (the point of this entry point is a caller that
// must not block on locks other threads hold); only the one-time look-up is serialised.
// A cudaDeviceReset invalidates the cached address: this entry point must not be used on
// that device again in the process afterwards.
std::mutex g_setup_mutex;
std::atomic<TopkRec*> g_scratch_ptr[kMaxDevices] = {};

// Device address of the scratch on the current device, looked up once per device.
mcd_status scratch_for_current_device(TopkRec** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return MCD_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return MCD_ERR_UNSUPPORTED;
  TopkRec* ptr = g_scratch_ptr[dev].load(std::memory_order_acquire);
  if (!ptr) {
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    ptr = g_scratch_ptr[dev].load(std::memory_order_relaxed);
    if (!ptr) {
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_topk_scratch) != cudaSuccess || !p) return MCD_ERR_CUDA;
      ptr = static_cast<TopkRec*>(p);
      g_scratch_ptr[dev].store(ptr, std::memory_order_release);
    }
  }
  *out = ptr;
  return MCD_OK;
}

// One CTA of 256 threads per row: the record goes to the static scratch, then the listed
// ids / weights / sum are copied to the caller's buffers.
__global__ void __launch_bounds__(kConsumerThreads)
    topk_rows_static_kernel(const float* logits, int V, int k, float T, TopkRec* recs, int32_t* ids,
                            uint32_t* weights, unsigned long long* sums) {
  __shared__ __align__(16) uint8_t smem_raw[sizeof(TopkScratch)];
  TopkScratch& ts = *reinterpret_cast<TopkScratch*>(smem_raw);
  const int row = blockIdx.x;
  TopkRec* r = recs + row;
  block_topk(logits + (size_t)row * V, V, k, T, 0, ts, r);
  consumer_sync();
  __threadfence_block();
  for (int i = threadIdx.x; i < k; i += kConsumerThreads) {
    if (ids) ids[(size_t)row * k + i] = r->ids[i];
    if (weights) weights[(size_t)row * k + i] = r->W[i];
  }
  if (threadIdx.x == 0 && sums) sums[row] = r->S;
}

}  // namespace
}  // namespace mcd

using namespace mcd;

extern "C" mcd_status mcd_topk_softmax_static(int32_t n_rows, int32_t vocab, int32_t top_k, float temperature,
                                              const float* logits, int32_t* ids, uint32_t* weights,
                                              uint64_t* sums, void* cuda_stream) {
  if (n_rows < 0 || !logits) return MCD_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(logits) & 15u) return MCD_ERR_INVALID_ARG;   // 16-byte row loads
  if (vocab < 16 || vocab % 16 || top_k < 1 || top_k > vocab) return MCD_ERR_INVALID_ARG;
  if (!(temperature > 0.f) || !std::isfinite(temperature)) return MCD_ERR_INVALID_ARG;
  if (vocab > kMaxVocab || top_k > kMaxTopK || n_rows > kStaticTopkRows) return MCD_ERR_UNSUPPORTED;
  TopkRec* scratch = nullptr;
  const mcd_status s = scratch_for_current_device(&scratch);   // first call per device: set-up
  if (s != MCD_OK) return s;
  if (n_rows == 0) return MCD_OK;
  topk_rows_static_kernel<<<n_rows, kConsumerThreads, 0, static_cast<cudaStream_t>(cuda_stream)>>>(
      logits, vocab, top_k, temperature, scratch, ids, weights, reinterpret_cast<unsigned long long*>(sums));
  return cudaGetLastError() == cudaSuccess ? MCD_OK : MCD_ERR_CUDA;
}
