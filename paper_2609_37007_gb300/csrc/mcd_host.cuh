// Host-side helpers shared by the library's API translation units (not part of the C ABI):
// weight re-tiling into units, geometry, norm conversion and access to an inner context.
#pragma once
#include <cstdio>
#include <cstdlib>

#include "mcd_internal.cuh"

namespace mcd {

// Source rows of one tiled matrix: up to three row-major segments stacked (Q, K, V), or the
// gate / up pair interleaved per 8 rows.
struct RowSrc {
  const uint8_t* seg[3];
  int seg_rows[3];
  int nseg;
  int interleave_gu;  // 1: logical tile t = [gate rows 8t..8t+7 ; up rows 8t..8t+7]
  int src_cols;       // elements per source row
};

// Logical element (r, c) -> offset (in elements) inside the tiled matrix.
__host__ __device__ inline long long tiled_offset(const MatGeom& g, int r, int c, int wdtype) {
  const int kc = c / (g.Ku * 16), kt = (c % (g.Ku * 16)) / 16;
  const int mb = r / (g.Mu * 16), mi = (r % (g.Mu * 16)) / 16;
  const long long u = (long long)kc * g.n_mb + mb;
  const long long tile = (u * g.Mu + mi) * g.Ku + kt;
  const int rr = r & 15, cc = c & 15;
  int pos;
  if (wdtype != MCD_WEIGHT_F32) {          // bf16 / int8: mma.m16n8k16 A-fragment order
    const int lane = (rr & 7) * 4 + ((cc & 7) >> 1);
    const int reg = (rr >> 3) + 2 * (cc >> 3);
    pos = lane * 8 + reg * 2 + (cc & 1);
  } else {
    pos = (rr + 16 * (cc >> 3)) * 8 + (cc & 7);
  }
  return tile * 256 + pos;
}

// Re-tile a row-major matrix (source elements: fp32 for MCD_WEIGHT_F32, else bf16); for
// MCD_WEIGHT_INT8 the elements are quantised with the per-row `scale` (see row_scale_kernel).
__global__ void tile_kernel(RowSrc rs, MatGeom g, int wdtype, uint8_t* dst, const float* scale);
// W8A16 row scales of a matrix in tiled row order: scale[r] = fp32(max |w_r| / 127).
__global__ void row_scale_kernel(RowSrc rs, MatGeom g, float* scale);
__global__ void to_f32_kernel(const uint8_t* src, int wdtype, long long n, float* dst);
// (cos, sin) of position pos and frequency i for pos < n_pos: [n_pos][D/2].
__global__ void rope_kernel(float2* rope, int D, double base, int n_pos);

bool make_geom(int M, int K, int Mu, int tile_bytes, int max_cols, MatGeom& g);
// Unit geometry of the backbone matrices and of an LM head with `head_rows` outputs.
bool backbone_geom(FrameParams& p, int head_rows);

// Device copies of one layer's source tensors (row-major, weight dtype); W8A16 scale arrays
// of the layer (null unless MCD_WEIGHT_INT8).
struct LayerSrc {
  const uint8_t *wq, *wk, *wv, *wo, *wg, *wu, *wd, *attn_norm, *ffn_norm, *q_norm, *k_norm;
};
// Re-tile layer l into p's weight arrays and convert its norm gains.
void load_layer(const FrameParams& p, cudaStream_t stream, const LayerSrc& src, int l);

mcd_status cuda_status(cudaError_t e);

// Batched decoding of many streams (GEMM path, mcd_batch.cu).
struct BatchState;
int batch_rows(const FrameParams& p, int max_streams);
constexpr int kBatchMinStreams = 5;
// Launches of this many streams go to the batched path even when the frame kernel fits them.
bool batch_prefers(const FrameParams& p, int n_streams);
mcd_status batch_create(const FrameParams& p, int max_streams, BatchState** out);
// The batched path's copies of layer l's weights for its tensor-core GEMMs (no-op without).
mcd_status batch_load_layer(BatchState* bs, const FrameParams& p, cudaStream_t st, const LayerSrc& src, int l);
mcd_status batch_load_head(BatchState* bs, const FrameParams& p, cudaStream_t st, const uint8_t* src, int P);
void batch_destroy(BatchState* bs);
mcd_status batch_decode(BatchState* bs, const FrameParams& p, cudaStream_t stream, int n, const uint32_t* stream_ids,
                        const uint32_t* frame_ids, const float* cond, const int32_t* c0, const float* c0_emb,
                        int32_t* codes_out, mcd_frame_stats* stats, uint8_t* trace);

// The inner (MultiCodeDecoder) context's parameters and stream.
const FrameParams& ctx_params(const mcd_ctx* c);
cudaStream_t ctx_stream(const mcd_ctx* c);
bool ctx_weights_loaded(const mcd_ctx* c);

}  // namespace mcd

#define MCD_CHECK(call)                                                                                  \
  do {                                                                                                   \
    cudaError_t e__ = (call);                                                                            \
    if (e__ != cudaSuccess) {                                                                            \
      if (getenv("MCD_DEBUG"))                                                                           \
        fprintf(stderr, "mcd: %s failed: %s (%s:%d)\n", #call, cudaGetErrorString(e__), __FILE__, __LINE__); \
      return mcd::cuda_status(e__);                                                                      \
    }                                                                                                    \
  } while (0)
