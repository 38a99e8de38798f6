// C ABI of libmcd (declared in include/mcd.h): context management, weight loading and
// re-tiling, frame decoding through the persistent frame kernel, the stepwise API and
// the sampler parity hooks.
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <string>
#include <vector>

#include "mcd_internal.cuh"
#include "mcd_sampler.cuh"
#include "mcd_host.cuh"

namespace mcd {
cudaError_t launch_frame_kernel(const FrameParams& p, cudaStream_t stream);
cudaError_t prepare_frame_kernel(int* max_ctas_per_sm);
int frame_smem_bytes();

// ------------------------------------------------------------------------------------
// Auxiliary kernels
// ------------------------------------------------------------------------------------
// Source row of tiled row r.
__device__ inline const uint8_t* src_row(const RowSrc& rs, int r, int es) {
  const uint8_t* src;
  int sr;
  if (rs.interleave_gu) {
    const int t = r >> 4, rr = r & 15;
    src = rs.seg[rr < 8 ? 0 : 1];
    sr = 8 * t + (rr & 7);
  } else {
    int rem = r, s = 0;
    while (s < rs.nseg - 1 && rem >= rs.seg_rows[s]) rem -= rs.seg_rows[s++];
    src = rs.seg[s];
    sr = rem;
  }
  return src + (long long)sr * rs.src_cols * es;
}

// W8A16 quantisation of one element: q = clamp(rint(fp32(w / s)), -127, 127), 0 if s = 0.
__device__ inline int quantise_w8(float w, float s) {
  if (!(s > 0.f)) return 0;
  const float q = rintf(__fdiv_rn(w, s));
  return (int)fminf(127.f, fmaxf(-127.f, q));
}

__global__ void tile_kernel(RowSrc rs, MatGeom g, int wdtype, uint8_t* dst, const float* scale) {
  const long long total = (long long)g.M * g.K;
  const int es = wdtype == MCD_WEIGHT_F32 ? 4 : 2;                        // source element bytes
  const int ed = wdtype == MCD_WEIGHT_F32 ? 4 : (wdtype == MCD_WEIGHT_INT8 ? 1 : 2);   // tiled element bytes
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < total;
       e += (long long)gridDim.x * blockDim.x) {
    const int r = (int)(e / g.K), c = (int)(e % g.K);
    const uint8_t* src = src_row(rs, r, es) + (long long)c * es;
    const long long d = tiled_offset(g, r, c, wdtype) * ed;
    if (ed == 1) {
      const float w = bf16_bits_to_f32(*reinterpret_cast<const uint16_t*>(src));
      reinterpret_cast<int8_t*>(dst)[d] = (int8_t)quantise_w8(w, scale[r]);
    } else if (ed == 2) {
      *reinterpret_cast<uint16_t*>(dst + d) = *reinterpret_cast<const uint16_t*>(src);
    } else {
      *reinterpret_cast<uint32_t*>(dst + d) = *reinterpret_cast<const uint32_t*>(src);
    }
  }
}

// One warp per tiled row: s = fp32(max |w| / 127) over the row's bf16 source values.
__global__ void row_scale_kernel(RowSrc rs, MatGeom g, float* scale) {
  const int r = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (r >= g.M) return;
  const uint16_t* src = reinterpret_cast<const uint16_t*>(src_row(rs, r, 2));
  float m = 0.f;
  for (int c = lane; c < g.K; c += 32) m = fmaxf(m, fabsf(bf16_bits_to_f32(src[c])));
  for (int o = 16; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
  if (lane == 0) scale[r] = __fdiv_rn(m, 127.f);
}

__global__ void to_f32_kernel(const uint8_t* src, int wdtype, long long n, float* dst) {
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x)
    dst[i] = wdtype != MCD_WEIGHT_F32 ? bf16_bits_to_f32(reinterpret_cast<const uint16_t*>(src)[i])
                                       : reinterpret_cast<const float*>(src)[i];
}

// LMH_P b_j for j = 1..K from the row-major head (one warp per output): the offsets'
// additive share of the draft logits, LMH_P (h + b_j) = LMH_P h + LMH_P b_j.
__global__ void head_bias_kernel(const uint8_t* head, const float* offsets, int K, int V, int H, int wdtype,
                                 const float* scale, float* out) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (warp >= K * V) return;
  const int j = warp / V, id = warp % V;
  float acc = 0.f;
  for (int k = lane; k < H; k += 32) {
    float w = wdtype != MCD_WEIGHT_F32 ? bf16_bits_to_f32(reinterpret_cast<const uint16_t*>(head)[(size_t)id * H + k])
                                       : reinterpret_cast<const float*>(head)[(size_t)id * H + k];
    if (wdtype == MCD_WEIGHT_INT8) w = (float)quantise_w8(w, scale[id]) * scale[id];   // the W8A16 head's value
    acc += w * offsets[(size_t)j * H + k];
  }
  for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, o);
  if (lane == 0) out[(size_t)j * V + id] = acc;
}

__global__ void rope_kernel(float2* rope, int D, double base, int n_pos) {
  const int half = D / 2;
  for (int idx = blockIdx.x * blockDim.x + threadIdx.x; idx < n_pos * half; idx += gridDim.x * blockDim.x) {
    const int pos = idx / half, i = idx % half;
    const double ang = (double)pos * pow(base, -2.0 * (double)i / (double)D);
    rope[idx] = make_float2((float)cos(ang), (float)sin(ang));
  }
}

__global__ void begin_frame_kernel(DevState* sts, unsigned* ctr, int n_ctr, const int* c0, int C0V, int S) {
  for (int i = threadIdx.x; i < n_ctr; i += blockDim.x) ctr[i] = 0u;
  if (threadIdx.x < S) init_stream_state(sts + threadIdx.x, C0V > 0 ? c0[threadIdx.x] : -1);
}

// Reset counters of a single stepwise call (the call index of the state).
// Counters of the slots one stepwise launch can use (a verify call, its noisy-target
// drafting passes, and the next slot whose ready flag it raises).
__global__ void reset_call_counters_kernel(const DevState* st, unsigned* ctr, int stride) {
  const int first = st->call;
  for (int sl = first; sl < min(first + kMaxDraft + 2, kMaxSlots); ++sl)
    for (int i = threadIdx.x; i < stride; i += blockDim.x) ctr[sl * stride + i] = 0u;
}

__global__ void zero_emitted_kernel(const DevState* st, int* n_emitted) {
  if (threadIdx.x == 0 && st->done && n_emitted) *n_emitted = 0;
}

// Top-k of n rows (one CTA of 256 threads per row).
__global__ void __launch_bounds__(kConsumerThreads) topk_rows_kernel(const float* logits, int V, int k, float T,
                                                                     TopkRec* recs, int32_t* ids, uint32_t* weights,
                                                                     unsigned long long* sums) {
  extern __shared__ __align__(16) uint8_t smem_raw[];
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

// Acceptance on given logits: rows 0..n_d of p, rows 0..n_d-1 of q, one CTA.
__global__ void __launch_bounds__(kConsumerThreads) accept_logits_kernel(FrameParams p, int a, int n_d, int call,
                                                                         const float* pl, const float* ql,
                                                                         const int* draft_ids, TopkRec* recs,
                                                                         int* emitted, int* out2) {
  extern __shared__ __align__(16) uint8_t smem_raw[];
  TopkScratch& ts = *reinterpret_cast<TopkScratch*>(smem_raw);
  const int n_p = (a + 1 + n_d <= p.P) ? n_d + 1 : n_d;
  for (int i = 0; i < n_p; ++i) {
    block_topk(pl + (size_t)i * p.V, p.V, p.top_k, p.T, 0, ts, recs + i);
    consumer_sync();
  }
  for (int i = 0; i < n_d; ++i) {
    block_topk(ql + (size_t)i * p.V, p.V, p.top_k, p.T, p.draft_mode == MCD_DRAFT_GREEDY, ts,
               recs + kMaxRows + i);
    consumer_sync();
  }
  __threadfence();
  consumer_sync();
  if (threadIdx.x < 32) {
    int drafts[kMaxDraft + 1];
    for (int i = 0; i < n_d; ++i) drafts[i] = draft_ids[i];
    AcceptResult r = warp_accept(
        a, n_d, p.P, drafts, [&](int i) { return (const TopkRec*)(recs + i); },
        [&](int i) { return (const TopkRec*)(recs + kMaxRows + i); }, p.seed, p.stream_ids[0], p.frame_ids[0], call);
    if (threadIdx.x == 0) {
      for (int t = 0; t < r.n_emit; ++t) emitted[t] = r.emitted[t];
      out2[0] = r.n_acc;
      out2[1] = r.n_emit;
    }
  }
}

// Draft logits z_j = LMH_{k+j}(h + b_j), one warp per (j, output id), from tiled heads.
__global__ void draft_logits_kernel(FrameParams p, int pos_k, int n_j, const float* h, float* z) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5, lane = threadIdx.x & 31;
  if (warp >= n_j * p.V) return;
  const int j = warp / p.V + 1, id = warp % p.V;
  const MatGeom& g = p.g[MAT_HEAD];
  const uint8_t* W = p.w_head + (long long)(pos_k + j - 1) * g.stride;
  float acc = 0.f;
  for (int k = lane; k < p.H; k += 32) {
    const long long off = tiled_offset(g, id, k, p.wdtype);
    const float w = p.wdtype == MCD_WEIGHT_BF16   ? bf16_bits_to_f32(reinterpret_cast<const uint16_t*>(W)[off])
                    : p.wdtype == MCD_WEIGHT_INT8 ? (float)reinterpret_cast<const int8_t*>(W)[off] *
                                                        p.s_head[(size_t)(pos_k + j - 1) * p.V + id]
                                                  : reinterpret_cast<const float*>(W)[off];
    acc += w * (h[k] + p.offsets[(size_t)(j - 1) * p.H + k]);
  }
  for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xFFFFFFFFu, acc, o);
  if (lane == 0) z[(size_t)(j - 1) * p.V + id] = acc;
}

__global__ void __launch_bounds__(kConsumerThreads) draft_sample_kernel(FrameParams p, int pos_k, int call,
                                                                        const float* z, TopkRec* recs, int* draft_ids,
                                                                        int* q_ids, uint32_t* q_weights) {
  extern __shared__ __align__(16) uint8_t smem_raw[];
  TopkScratch& ts = *reinterpret_cast<TopkScratch*>(smem_raw);
  const int j = blockIdx.x + 1;
  TopkRec* r = recs + blockIdx.x;
  block_topk(z + (size_t)(j - 1) * p.V, p.V, p.top_k, p.T, p.draft_mode == MCD_DRAFT_GREEDY, ts, r);
  consumer_sync();
  __threadfence_block();
  if (threadIdx.x < 32) {
    const unsigned long long U = uniform_U(p.seed, p.stream_ids[0], p.frame_ids[0], call, pos_k + j, PURPOSE_DRAFT);
    const int d = warp_draw(r, U);
    if (threadIdx.x == 0) draft_ids[j - 1] = d;
  }
  for (int i = threadIdx.x; i < p.top_k; i += kConsumerThreads) {
    if (q_ids) q_ids[(size_t)(j - 1) * p.top_k + i] = i < r->n ? r->ids[i] : -1;
    if (q_weights) q_weights[(size_t)(j - 1) * p.top_k + i] = i < r->n ? r->W[i] : 0u;
  }
}

}  // namespace mcd

using namespace mcd;

// ------------------------------------------------------------------------------------
// Context
// ------------------------------------------------------------------------------------
struct mcd_ctx {
  mcd_config cfg;
  cudaStream_t stream;
  int device;
  FrameParams fp;
  std::vector<void*> allocs;
  uint8_t* w_arena = nullptr;
  size_t w_bytes = 0;
  size_t off_qkv = 0, off_wo = 0, off_gu = 0, off_wd = 0, off_head = 0, off_embed = 0;
  float* f32_arena = nullptr;   // norms + offsets
  uint8_t* host_stage = nullptr;  // device staging for mcd_decode_frame_host (holds the err word)
  uint8_t* host_pin = nullptr;    // pinned host mirror of host_stage
  bool weights_loaded = false;
  bool frame_begun = false;
  int h_err = 0;                 // host-side sticky CUDA error
  mcd::BatchState* batch = nullptr;   // GEMM path for calls with more than kMaxCols packed rows
};

mcd_status mcd::cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return MCD_OK;
  if (e == cudaErrorMemoryAllocation) return MCD_ERR_OOM;
  return MCD_ERR_CUDA;
}

const FrameParams& mcd::ctx_params(const mcd_ctx* c) { return c->fp; }
cudaStream_t mcd::ctx_stream(const mcd_ctx* c) { return c->stream; }
bool mcd::ctx_weights_loaded(const mcd_ctx* c) { return c->weights_loaded; }

template <class T>
static cudaError_t ctx_alloc(mcd_ctx* c, T** p, size_t bytes) {
  void* q = nullptr;
  cudaError_t e = cudaMalloc(&q, bytes < 256 ? 256 : bytes);
  if (e != cudaSuccess) return e;
  c->allocs.push_back(q);
  *p = static_cast<T*>(q);
  return cudaSuccess;
}

bool mcd::make_geom(int M, int K, int Mu, int tile_bytes, int max_cols, MatGeom& g) {
  const int Gk = kConsumerWarps / Mu;
  if (M % (Mu * 16) || K % 16) return false;
  const int kt = K / 16;
  int Ku = 0;
  for (int cand = kt; cand >= Gk; --cand) {
    if (kt % cand == 0 && cand % Gk == 0 && Mu * cand * tile_bytes <= kSlotBytes && cand * 16 <= max_cols) {
      Ku = cand;
      break;
    }
  }
  if (!Ku) return false;
  g.M = M;
  g.K = K;
  g.Mu = Mu;
  g.Ku = Ku;
  g.n_mb = M / (Mu * 16);
  g.n_kc = kt / Ku;
  g.n_units = g.n_mb * g.n_kc;
  g.unit_bytes = Mu * Ku * tile_bytes;
  g.stride = (long long)g.n_units * g.unit_bytes;
  return true;
}

bool mcd::backbone_geom(FrameParams& p, int head_rows) {
  // bytes per 16 x 16 tile; one-byte W8A16 tiles go two m-tiles per unit to keep units at 32 KB
  const int tb = p.wdtype == MCD_WEIGHT_BF16 ? 512 : p.wdtype == MCD_WEIGHT_INT8 ? 256 : 1024;
  const int mu = p.wdtype == MCD_WEIGHT_INT8 ? 2 : 1;
  auto mu_for = [&](int rows) { return rows % (mu * 16) == 0 ? mu : 1; };
  bool ok = make_geom(p.qkv_dim, p.H, mu_for(p.qkv_dim), tb, 1024, p.g[MAT_QKV]) && p.g[MAT_QKV].n_kc == 1;
  int mu_o = 8;
  while (mu_o > 1 && (mu_o * (p.D / 16) * tb > kSlotBytes || p.H % (mu_o * 16))) mu_o >>= 1;
  ok = ok && make_geom(p.H, p.NH * p.D, mu_o, tb, p.D, p.g[MAT_WO]) && p.g[MAT_WO].Ku * 16 == p.D;
  ok = ok && make_geom(2 * p.F, p.H, mu_for(2 * p.F), tb, 1024, p.g[MAT_GU]) && p.g[MAT_GU].n_kc == 1;
  ok = ok && make_geom(p.H, p.F, mu_for(p.H), tb, 1024, p.g[MAT_WD]);
  // (heads keep one m-tile per unit: the draft-offset bias tiles are staged per 16 rows)
  ok = ok && make_geom(head_rows, p.H, 1, tb, 1024, p.g[MAT_HEAD]) && p.g[MAT_HEAD].n_kc == 1;
  return ok;
}

void mcd::load_layer(const FrameParams& p, cudaStream_t stream, const LayerSrc& src, int l) {
  const int H = p.H, D = p.D, F = p.F, qd = p.NH * D, kd = p.NKV * D;
  const bool q8 = p.wdtype == MCD_WEIGHT_INT8;
  auto tile = [&](RowSrc rs, const MatGeom& g, const uint8_t* dst, const float* scale) {
    float* sc = const_cast<float*>(scale);
    if (q8) row_scale_kernel<<<(g.M * 32 + 255) / 256, 256, 0, stream>>>(rs, g, sc);
    tile_kernel<<<1024, 256, 0, stream>>>(rs, g, p.wdtype, const_cast<uint8_t*>(dst), q8 ? sc : nullptr);
  };
  auto conv = [&](const uint8_t* from, int64_t count, const float* dst) {
    to_f32_kernel<<<64, 256, 0, stream>>>(from, p.wdtype, count, const_cast<float*>(dst));
  };
  RowSrc rs{};
  rs.seg[0] = src.wq;
  rs.seg[1] = src.wk;
  rs.seg[2] = src.wv;
  rs.seg_rows[0] = qd;
  rs.seg_rows[1] = kd;
  rs.seg_rows[2] = kd;
  rs.nseg = 3;
  rs.src_cols = H;
  tile(rs, p.g[MAT_QKV], p.w_qkv + (size_t)l * p.g[MAT_QKV].stride, q8 ? p.s_qkv + (size_t)l * p.qkv_dim : nullptr);
  RowSrc ro{};
  ro.seg[0] = src.wo;
  ro.seg_rows[0] = H;
  ro.nseg = 1;
  ro.src_cols = qd;
  tile(ro, p.g[MAT_WO], p.w_wo + (size_t)l * p.g[MAT_WO].stride, q8 ? p.s_wo + (size_t)l * H : nullptr);
  RowSrc rg{};
  rg.seg[0] = src.wg;
  rg.seg[1] = src.wu;
  rg.nseg = 2;
  rg.interleave_gu = 1;
  rg.src_cols = H;
  tile(rg, p.g[MAT_GU], p.w_gu + (size_t)l * p.g[MAT_GU].stride, q8 ? p.s_gu + (size_t)l * 2 * F : nullptr);
  RowSrc rd{};
  rd.seg[0] = src.wd;
  rd.seg_rows[0] = H;
  rd.nseg = 1;
  rd.src_cols = F;
  tile(rd, p.g[MAT_WD], p.w_wd + (size_t)l * p.g[MAT_WD].stride, q8 ? p.s_wd + (size_t)l * H : nullptr);
  conv(src.attn_norm, H, p.attn_norm + (size_t)l * H);
  conv(src.ffn_norm, H, p.ffn_norm + (size_t)l * H);
  if (p.qk_norm) {
    conv(src.q_norm, D, p.q_norm + (size_t)l * D);
    conv(src.k_norm, D, p.k_norm + (size_t)l * D);
  }
}

static mcd_status validate_config(const mcd_config& c) {
  if (c.n_layers < 1 || c.hidden < 128 || c.hidden % 128 || c.hidden > 1024) return MCD_ERR_UNSUPPORTED;
  if (!(c.head_dim == 64 || c.head_dim == 128)) return MCD_ERR_UNSUPPORTED;
  if (c.n_q_heads < 1 || c.n_kv_heads < 1 || c.n_q_heads % c.n_kv_heads) return MCD_ERR_INVALID_ARG;
  if (c.ffn < 128 || c.ffn % 128) return MCD_ERR_UNSUPPORTED;
  if (c.n_pos < 1 || c.n_pos > 15) return MCD_ERR_UNSUPPORTED;
  if (c.vocab < 16 || c.vocab % 16 || c.vocab > kMaxVocab) return MCD_ERR_UNSUPPORTED;
  if (c.c0_vocab < 0 || c.c0_vocab > kMaxVocab) return MCD_ERR_UNSUPPORTED;
  if (c.draft_len < 0 || c.draft_len > kMaxDraft) return MCD_ERR_UNSUPPORTED;
  if (c.top_k < 1 || c.top_k > kMaxTopK || c.top_k > c.vocab) return MCD_ERR_UNSUPPORTED;
  if (!(c.temperature > 0.f) || !(c.rms_eps > 0.f) || !(c.rope_base > 1.f)) return MCD_ERR_INVALID_ARG;
  if (c.weight_dtype < MCD_WEIGHT_F32 || c.weight_dtype > MCD_WEIGHT_INT8) return MCD_ERR_INVALID_ARG;
  if (c.draft_mode < 0 || c.draft_mode > MCD_DRAFT_TREE) return MCD_ERR_INVALID_ARG;
  if (c.draft_mode == MCD_DRAFT_TREE && (c.max_streams != 1 || c.draft_len < 1)) return MCD_ERR_UNSUPPORTED;
  if (c.draft_mode == MCD_DRAFT_NOISY_TARGET && !(c.noise_sigma >= 0.f)) return MCD_ERR_INVALID_ARG;
  if (c.max_streams < 1 || c.max_streams > kMaxBatchStreams) return MCD_ERR_UNSUPPORTED;
  if (c.max_streams > 1 && c.draft_mode == MCD_DRAFT_NOISY_TARGET) return MCD_ERR_UNSUPPORTED;
  // beyond kMaxCols packed rows per call (or kMaxStreams streams) calls run on the batched
  // GEMM path: bf16 weights, at most kMaxBatchRows rows, 16 query vectors per (stream, KV head)
  const int rows = c.max_streams * std::max(c.draft_len + 1, 2);
  if (rows > kMaxCols || c.max_streams > kMaxStreams) {
    if (c.weight_dtype != MCD_WEIGHT_BF16 || rows > kMaxBatchRows) return MCD_ERR_UNSUPPORTED;
    if (std::max(c.draft_len + 1, 2) * (c.n_q_heads / c.n_kv_heads) > 16) return MCD_ERR_UNSUPPORTED;
  }
  if ((long long)c.n_q_heads * c.head_dim + 2LL * c.n_kv_heads * c.head_dim > 8192) return MCD_ERR_UNSUPPORTED;
  return MCD_OK;
}

extern "C" {

const char* mcd_status_str(mcd_status s) {
  switch (s) {
    case MCD_OK: return "ok";
    case MCD_ERR_INVALID_ARG: return "invalid argument";
    case MCD_ERR_STATE: return "call out of order";
    case MCD_ERR_CUDA: return "CUDA error";
    case MCD_ERR_OOM: return "out of device memory";
    case MCD_ERR_TIMEOUT: return "device-side wait timed out";
    case MCD_ERR_WEIGHTS: return "missing or malformed weight tensor";
    case MCD_ERR_UNSUPPORTED: return "shape outside the kernels' limits";
  }
  return "unknown status";
}

// Staging area of mcd_decode_frame_host, mirrored in pinned host memory:
//   cond [H] | c0 (16 B) | c0_emb [H] | codes [n_pos <= 15] (64 B) | stats (32 B) | err (16 B).
// The inputs are one contiguous H2D range and the results plus the device error word one
// contiguous D2H range, so a host-buffer frame costs two copies and one stream wait.
static size_t stage_cond(const FrameParams&) { return 0; }
static size_t stage_c0(const FrameParams& p) { return (size_t)p.H * 4; }
static size_t stage_emb(const FrameParams& p) { return (size_t)p.H * 4 + 16; }
static size_t stage_codes(const FrameParams& p) { return (size_t)p.H * 8 + 16; }
static size_t stage_stats(const FrameParams& p) { return stage_codes(p) + 64; }
static size_t stage_err(const FrameParams& p) { return stage_stats(p) + 32; }
static size_t host_stage_bytes(const FrameParams& p) { return stage_err(p) + 16; }
static_assert(sizeof(mcd_frame_stats) <= 32, "stats slot of the staging area");

mcd_status mcd_create(const mcd_config* cfg, void* cuda_stream, mcd_ctx** out) {
  if (!out) return MCD_ERR_INVALID_ARG;
  *out = nullptr;
  if (!cfg) return MCD_ERR_INVALID_ARG;
  mcd_status vs = validate_config(*cfg);
  if (vs != MCD_OK) return vs;
  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || ndev == 0) return MCD_ERR_CUDA;
  mcd_ctx* c = new mcd_ctx();
  c->cfg = *cfg;
  c->stream = static_cast<cudaStream_t>(cuda_stream);
  auto fail = [&](mcd_status s) {
    mcd_destroy(c);
    return s;
  };
  if (cudaGetDevice(&c->device) != cudaSuccess) return fail(MCD_ERR_CUDA);
  int n_sm = 0, coop = 0, max_blocks = 0;
  if (cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, c->device) != cudaSuccess) return fail(MCD_ERR_CUDA);
  if (cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, c->device) != cudaSuccess || !coop)
    return fail(MCD_ERR_UNSUPPORTED);
  if (prepare_frame_kernel(&max_blocks) != cudaSuccess || max_blocks < 1) return fail(MCD_ERR_UNSUPPORTED);

  const mcd_config& k = *cfg;
  FrameParams& p = c->fp;
  memset(&p, 0, sizeof(p));
  p.L = k.n_layers;
  p.H = k.hidden;
  p.NH = k.n_q_heads;
  p.NKV = k.n_kv_heads;
  p.D = k.head_dim;
  p.F = k.ffn;
  p.P = k.n_pos;
  p.V = k.vocab;
  p.C0V = k.c0_vocab;
  p.K = k.draft_len;
  p.top_k = k.top_k;
  p.qk_norm = k.qk_norm;
  p.wdtype = k.weight_dtype;
  p.draft_mode = k.draft_mode;
  p.eps = k.rms_eps;
  p.T = k.temperature;
  p.sigma = k.noise_sigma;
  p.seed = k.seed;
  p.qkv_dim = p.NH * p.D + 2 * p.NKV * p.D;
  p.n_cta = n_sm;
  p.wait_ns = 2000000000ull;  // 2 s
  p.S = 1;
  p.trace_stride = (long long)sizeof(mcd_call_trace) * kMaxCalls + (long long)2 * kMaxCalls * kMaxRows * p.V * 4;
  if (k.draft_mode == MCD_DRAFT_TREE)   // + the tree records and every row's verify logits
    p.trace_stride += (long long)sizeof(mcd_tree_trace) * kMaxCalls + (long long)kMaxCalls * kMaxTreeRows * p.V * 4;
  // MCD_WAIT_NS overrides the bound, never below 100 ms: the same bound limits how long an
  // aborting CTA waits for its copies and MMAs in flight, which must land before it exits.
  const char* wn = getenv("MCD_WAIT_NS");
  if (wn) p.wait_ns = std::max(strtoull(wn, nullptr, 10), 100000000ull);

  const int es = k.weight_dtype == MCD_WEIGHT_F32 ? 4 : 2;     // embedding tables (bf16 for W8A16)
  const bool ok = backbone_geom(p, p.V);
  if (!ok) return fail(MCD_ERR_UNSUPPORTED);
  p.ctr_stride = ctr_count(p.L);

  // weight arena
  const size_t sq = p.g[MAT_QKV].stride, so = p.g[MAT_WO].stride, sg = p.g[MAT_GU].stride, sd = p.g[MAT_WD].stride;
  c->off_qkv = 0;
  c->off_wo = c->off_qkv + sq * p.L;
  c->off_gu = c->off_wo + so * p.L;
  c->off_wd = c->off_gu + sg * p.L;
  c->off_head = c->off_wd + sd * p.L;
  c->off_embed = c->off_head + (size_t)p.g[MAT_HEAD].stride * p.P;
  p.embed_stride = (long long)std::max(p.C0V, p.V) * p.H * es;
  c->w_bytes = c->off_embed + (size_t)p.embed_stride * p.P;
  cudaError_t e;
  if ((e = ctx_alloc(c, &c->w_arena, c->w_bytes)) != cudaSuccess) return fail(cuda_status(e));
  p.w_qkv = c->w_arena + c->off_qkv;
  p.w_wo = c->w_arena + c->off_wo;
  p.w_gu = c->w_arena + c->off_gu;
  p.w_wd = c->w_arena + c->off_wd;
  p.w_head = c->w_arena + c->off_head;
  p.embed = c->w_arena + c->off_embed;

  const int Kd = std::max(p.K, 1);
  const size_t nf = (size_t)p.L * p.H * 2 + (size_t)p.L * p.D * 2 + p.H + (size_t)Kd * p.H;
  if ((e = ctx_alloc(c, &c->f32_arena, nf * 4)) != cudaSuccess) return fail(cuda_status(e));
  p.attn_norm = c->f32_arena;
  p.ffn_norm = p.attn_norm + (size_t)p.L * p.H;
  p.q_norm = p.ffn_norm + (size_t)p.L * p.H;
  p.k_norm = p.q_norm + (size_t)p.L * p.D;
  p.final_norm = p.k_norm + (size_t)p.L * p.D;
  p.offsets = p.final_norm + p.H;

  if (k.weight_dtype == MCD_WEIGHT_INT8) {    // W8A16 row scales
    const size_t ns = (size_t)p.L * (p.qkv_dim + 2 * p.H + 2 * p.F) + (size_t)p.P * p.V;
    float* sc = nullptr;
    if ((e = ctx_alloc(c, &sc, ns * 4)) != cudaSuccess) return fail(cuda_status(e));
    p.s_qkv = sc;
    p.s_wo = p.s_qkv + (size_t)p.L * p.qkv_dim;
    p.s_gu = p.s_wo + (size_t)p.L * p.H;
    p.s_wd = p.s_gu + (size_t)p.L * 2 * p.F;
    p.s_head = p.s_wd + (size_t)p.L * p.H;
  }
  float* head_bias = nullptr;
  if ((e = ctx_alloc(c, &head_bias, sizeof(float) * (size_t)p.P * Kd * p.V)) != cudaSuccess) return fail(cuda_status(e));
  p.head_bias = head_bias;
  float2* rope = nullptr;
  if ((e = ctx_alloc(c, &rope, sizeof(float2) * kMaxPos * (p.D / 2))) != cudaSuccess) return fail(cuda_status(e));
  p.rope = rope;
  if ((e = ctx_alloc(c, &p.x, sizeof(float) * kMaxCols * p.H)) != cudaSuccess) return fail(cuda_status(e));
  if ((e = ctx_alloc(c, &p.qkv, sizeof(float) * kMaxCols * p.qkv_dim)) != cudaSuccess) return fail(cuda_status(e));
  if ((e = ctx_alloc(c, &p.mbuf, sizeof(float) * kMaxCols * p.F)) != cudaSuccess) return fail(cuda_status(e));
  if ((e = ctx_alloc(c, &p.attn, sizeof(float) * kMaxCols * p.NH * p.D)) != cudaSuccess) return fail(cuda_status(e));
  if ((e = ctx_alloc(c, &p.logits, sizeof(float) * kMaxTreeRows * (kMaxDraft + 1) * p.V)) != cudaSuccess)
    return fail(cuda_status(e));
  // cache entries per (layer, KV head): the frame's positions, then in TREE mode the rows of
  // the current call (slot kMaxPos + row) until its acceptance step commits the kept ones
  p.kv_slots = kMaxPos + (k.draft_mode == MCD_DRAFT_TREE ? kMaxTreeRows : 0);
  p.kv_stride = (long long)p.L * p.NKV * p.kv_slots * p.D;
  const size_t kvsz = sizeof(float) * (size_t)p.kv_stride * k.max_streams;
  if ((e = ctx_alloc(c, &p.kcache, kvsz)) != cudaSuccess) return fail(cuda_status(e));
  if ((e = ctx_alloc(c, &p.vcache, kvsz)) != cudaSuccess) return fail(cuda_status(e));
  static_assert(kMaxTreeRows <= 2 * kMaxCols + 1, "record buffer rows");
  if ((e = ctx_alloc(c, &p.topk, sizeof(TopkRec) * (2 * kMaxCols + 1) * (kMaxDraft + 1))) != cudaSuccess)
    return fail(cuda_status(e));
  if ((e = ctx_alloc(c, &p.draftq, sizeof(TopkRec) * (kMaxDraft + 1))) != cudaSuccess) return fail(cuda_status(e));
  if ((e = ctx_alloc(c, &p.st, sizeof(DevState) * k.max_streams)) != cudaSuccess) return fail(cuda_status(e));
  if ((e = ctx_alloc(c, &p.ctr, sizeof(unsigned) * kMaxSlots * p.ctr_stride)) != cudaSuccess)
    return fail(cuda_status(e));
  if ((e = ctx_alloc(c, &c->host_stage, host_stage_bytes(p))) != cudaSuccess) return fail(cuda_status(e));
  p.err = reinterpret_cast<int*>(c->host_stage + stage_err(p));
  if ((e = cudaHostAlloc(reinterpret_cast<void**>(&c->host_pin), host_stage_bytes(p), cudaHostAllocDefault)) !=
      cudaSuccess) {
    c->host_pin = nullptr;
    return fail(cuda_status(e));
  }
  if ((e = ctx_alloc(c, &p.tree_cand, sizeof(int) * kMaxDraft * kMaxTreeRank)) != cudaSuccess)
    return fail(cuda_status(e));
  if (k.draft_mode == MCD_DRAFT_TREE) {       // until mcd_set_tree: the chain of K rank-0 nodes
    p.tree_n = k.draft_len;
    p.tree_maxd = k.draft_len;
    for (int i = 0; i < k.draft_len; ++i) {
      p.tree_parent[i] = (signed char)(i - 1);
      p.tree_rank[i] = 0;
      p.tree_depth[i] = (signed char)(i + 1);
      p.tree_m[i] = 1;
      p.tree_anc[i] = (2ull << i) - 1ull;
    }
  }
  if (cudaMemsetAsync(p.err, 0, sizeof(int), c->stream) != cudaSuccess) return fail(MCD_ERR_CUDA);
  if (cudaMemsetAsync(p.kcache, 0, kvsz, c->stream) != cudaSuccess) return fail(MCD_ERR_CUDA);
  if (cudaMemsetAsync(p.vcache, 0, kvsz, c->stream) != cudaSuccess) return fail(MCD_ERR_CUDA);
  if (cudaMemsetAsync(p.st, 0, sizeof(DevState) * k.max_streams, c->stream) != cudaSuccess) return fail(MCD_ERR_CUDA);
  rope_kernel<<<8, 256, 0, c->stream>>>(rope, p.D, (double)k.rope_base, kMaxPos);
  if (cudaGetLastError() != cudaSuccess) return fail(MCD_ERR_CUDA);
  if (cudaStreamSynchronize(c->stream) != cudaSuccess) return fail(MCD_ERR_CUDA);
  if (k.max_streams > kMaxStreams || batch_rows(p, k.max_streams) > kMaxCols || batch_prefers(p, k.max_streams)) {
    mcd_status bs = batch_create(p, k.max_streams, &c->batch);
    if (bs != MCD_OK) return fail(bs);
  }
  *out = c;
  return MCD_OK;
}

void mcd_destroy(mcd_ctx* c) {
  if (!c) return;
  cudaStreamSynchronize(c->stream);
  batch_destroy(c->batch);
  for (void* q : c->allocs) cudaFree(q);
  if (c->host_pin) cudaFreeHost(c->host_pin);
  delete c;
}

int32_t mcd_num_ctas(const mcd_ctx* c) { return c ? c->fp.n_cta : 0; }

int64_t mcd_call_weight_bytes(const mcd_ctx* c, int32_t n_heads) {
  if (!c) return 0;
  const FrameParams& p = c->fp;
  int64_t b = (int64_t)p.L * (p.g[MAT_QKV].stride + p.g[MAT_WO].stride + p.g[MAT_GU].stride + p.g[MAT_WD].stride) +
              (int64_t)n_heads * p.g[MAT_HEAD].stride;
  if (p.wdtype == MCD_WEIGHT_INT8)   // + the row scales the epilogues read
    b += 4LL * p.L * (p.qkv_dim + 2 * p.H + 2 * p.F) + 4LL * n_heads * p.V;
  return b;
}

mcd_status mcd_load_weights(mcd_ctx* c, int32_t n, const char* const* names, const void* const* host_ptrs,
                            const int64_t* nbytes) {
  if (!c || n <= 0 || !names || !host_ptrs || !nbytes) return MCD_ERR_INVALID_ARG;
  FrameParams& p = c->fp;
  const int es = p.wdtype == MCD_WEIGHT_F32 ? 4 : 2;           // source element bytes
  const int Kd = std::max(p.K, 1);
  std::map<std::string, std::pair<const void*, int64_t>> given;
  for (int i = 0; i < n; ++i) {
    if (!names[i] || !host_ptrs[i]) return MCD_ERR_INVALID_ARG;
    if (given.count(names[i])) return MCD_ERR_WEIGHTS;
    given[names[i]] = {host_ptrs[i], nbytes[i]};
  }
  // required tensors and their element counts
  std::vector<std::pair<std::string, int64_t>> req;
  const int64_t H = p.H, D = p.D, qd = (int64_t)p.NH * D, kd = (int64_t)p.NKV * D, F = p.F;
  for (int l = 0; l < p.L; ++l) {
    const std::string pre = "layers." + std::to_string(l) + ".";
    req.push_back({pre + "attn_norm", H});
    req.push_back({pre + "wq", qd * H});
    req.push_back({pre + "wk", kd * H});
    req.push_back({pre + "wv", kd * H});
    if (p.qk_norm) {
      req.push_back({pre + "q_norm", D});
      req.push_back({pre + "k_norm", D});
    }
    req.push_back({pre + "wo", H * qd});
    req.push_back({pre + "ffn_norm", H});
    req.push_back({pre + "wg", F * H});
    req.push_back({pre + "wu", F * H});
    req.push_back({pre + "wd", H * F});
  }
  req.push_back({"final_norm", H});
  if (p.C0V > 0) req.push_back({"embed.0", (int64_t)p.C0V * H});
  for (int i = 1; i < p.P; ++i) req.push_back({"embed." + std::to_string(i), (int64_t)p.V * H});
  for (int P = 1; P <= p.P; ++P) req.push_back({"head." + std::to_string(P), (int64_t)p.V * H});
  for (int j = 1; j <= Kd; ++j) req.push_back({"offset." + std::to_string(j), H});
  size_t stage_bytes = 0;
  std::map<std::string, size_t> soff;
  for (auto& r : req) {
    auto it = given.find(r.first);
    if (it == given.end() || it->second.second != r.second * es) {
      if (getenv("MCD_DEBUG")) fprintf(stderr, "mcd: weight %s missing or wrong size\n", r.first.c_str());
      return MCD_ERR_WEIGHTS;
    }
    soff[r.first] = stage_bytes;
    stage_bytes += (size_t)((it->second.second + 255) / 256 * 256);
  }
  uint8_t* stage = nullptr;
  MCD_CHECK(cudaMalloc(&stage, stage_bytes));
  auto cleanup = [&](mcd_status s) {
    cudaStreamSynchronize(c->stream);
    cudaFree(stage);
    return s;
  };
  for (auto& r : req) {
    auto& gv = given[r.first];
    if (cudaMemcpyAsync(stage + soff[r.first], gv.first, (size_t)gv.second, cudaMemcpyHostToDevice, c->stream) !=
        cudaSuccess)
      return cleanup(MCD_ERR_CUDA);
  }
  auto S = [&](const std::string& name) { return (const uint8_t*)(stage + soff[name]); };
  auto tile = [&](RowSrc rs, const MatGeom& g, uint8_t* dst, float* scale) {
    if (scale) row_scale_kernel<<<(g.M * 32 + 255) / 256, 256, 0, c->stream>>>(rs, g, scale);
    tile_kernel<<<1024, 256, 0, c->stream>>>(rs, g, p.wdtype, dst, scale);
  };
  const bool q8 = p.wdtype == MCD_WEIGHT_INT8;
  auto conv = [&](const std::string& name, int64_t count, const float* dst) {
    to_f32_kernel<<<64, 256, 0, c->stream>>>(S(name), p.wdtype, count, const_cast<float*>(dst));
  };
  for (int l = 0; l < p.L; ++l) {
    const std::string pre = "layers." + std::to_string(l) + ".";
    LayerSrc ls{S(pre + "wq"), S(pre + "wk"), S(pre + "wv"), S(pre + "wo"), S(pre + "wg"), S(pre + "wu"),
                S(pre + "wd"), S(pre + "attn_norm"), S(pre + "ffn_norm"),
                p.qk_norm ? S(pre + "q_norm") : nullptr, p.qk_norm ? S(pre + "k_norm") : nullptr};
    load_layer(p, c->stream, ls, l);
    if (c->batch && batch_load_layer(c->batch, p, c->stream, ls, l) != MCD_OK) return cleanup(MCD_ERR_CUDA);
  }
  conv("final_norm", H, p.final_norm);
  for (int j = 1; j <= Kd; ++j) conv("offset." + std::to_string(j), H, p.offsets + (size_t)(j - 1) * H);
  // LM heads (W8A16: row scales first, which the draft-offset biases also use)
  for (int P = 1; P <= p.P; ++P) {
    RowSrc rh{};
    rh.seg[0] = S("head." + std::to_string(P));
    rh.seg_rows[0] = p.V;
    rh.nseg = 1;
    rh.src_cols = (int)H;
    tile(rh, p.g[MAT_HEAD], c->w_arena + c->off_head + (size_t)(P - 1) * p.g[MAT_HEAD].stride,
         q8 ? const_cast<float*>(p.s_head) + (size_t)(P - 1) * p.V : nullptr);
    if (c->batch && batch_load_head(c->batch, p, c->stream, S("head." + std::to_string(P)), P) != MCD_OK)
      return cleanup(MCD_ERR_CUDA);
  }
  for (int P = 1; P <= p.P && p.K > 0; ++P) {
    const int warps = p.K * p.V;
    head_bias_kernel<<<(warps * 32 + 255) / 256, 256, 0, c->stream>>>(
        S("head." + std::to_string(P)), p.offsets, p.K, p.V, p.H, p.wdtype, q8 ? p.s_head + (size_t)(P - 1) * p.V : nullptr,
        const_cast<float*>(p.head_bias) + (size_t)(P - 1) * p.K * p.V);
  }
  if (p.C0V > 0)
    if (cudaMemcpyAsync(c->w_arena + c->off_embed, S("embed.0"), (size_t)p.C0V * H * es, cudaMemcpyDeviceToDevice,
                        c->stream) != cudaSuccess)
      return cleanup(MCD_ERR_CUDA);
  for (int i = 1; i < p.P; ++i)
    if (cudaMemcpyAsync(c->w_arena + c->off_embed + (size_t)i * p.embed_stride, S("embed." + std::to_string(i)),
                        (size_t)p.V * H * es, cudaMemcpyDeviceToDevice, c->stream) != cudaSuccess)
      return cleanup(MCD_ERR_CUDA);
  if (cudaGetLastError() != cudaSuccess) return cleanup(MCD_ERR_CUDA);
  mcd_status s = cleanup(MCD_OK);
  if (cudaGetLastError() != cudaSuccess) return MCD_ERR_CUDA;
  c->weights_loaded = true;
  return s;
}

static mcd_status launch_begin(mcd_ctx* c, int n, const uint32_t* stream_ids, const uint32_t* frame_ids,
                               const float* cond, const int32_t* c0, const float* c0_emb) {
  FrameParams& p = c->fp;
  if (!cond || n < 1 || !stream_ids || !frame_ids) return MCD_ERR_INVALID_ARG;
  if (n > c->cfg.max_streams) return MCD_ERR_INVALID_ARG;
  // the kernel reads these rows with 16-byte loads
  if ((reinterpret_cast<uintptr_t>(cond) & 15u) || (reinterpret_cast<uintptr_t>(c0_emb) & 15u))
    return MCD_ERR_INVALID_ARG;
  if (p.C0V > 0 && !c0) return MCD_ERR_INVALID_ARG;
  if (p.C0V == 0 && !c0_emb) return MCD_ERR_INVALID_ARG;
  p.cond = cond;
  p.c0 = c0;
  p.c0emb = c0_emb;
  p.S = n;
  for (int s = 0; s < kMaxStreams; ++s) {
    p.stream_ids[s] = s < n ? stream_ids[s] : 0u;
    p.frame_ids[s] = s < n ? frame_ids[s] : 0u;
  }
  begin_frame_kernel<<<1, 256, 0, c->stream>>>(p.st, p.ctr, kMaxSlots * p.ctr_stride, c0, p.C0V, n);
  MCD_CHECK(cudaGetLastError());
  c->frame_begun = true;
  return MCD_OK;
}

mcd_status mcd_decode_frames(mcd_ctx* c, int32_t n_streams, const uint32_t* stream_ids, const uint32_t* frame_idx,
                             const float* cond, const int32_t* c0, const float* c0_emb, int32_t* codes_out,
                             mcd_frame_stats* stats) {
  if (!c || !codes_out) return MCD_ERR_INVALID_ARG;
  if (!c->weights_loaded) return MCD_ERR_STATE;
  if (n_streams > kMaxStreams || batch_rows(c->fp, n_streams) > kMaxCols ||
      (c->batch && batch_prefers(c->fp, n_streams))) {
    // many streams: the batched GEMM path (one CUDA graph launch per frame)
    const FrameParams& p = c->fp;
    if (!c->batch || n_streams > c->cfg.max_streams) return MCD_ERR_INVALID_ARG;
    if (!cond || !stream_ids || !frame_idx) return MCD_ERR_INVALID_ARG;
    if (p.C0V > 0 && !c0) return MCD_ERR_INVALID_ARG;
    if (p.C0V == 0 && !c0_emb) return MCD_ERR_INVALID_ARG;
    c->frame_begun = false;
    return batch_decode(c->batch, p, c->stream, n_streams, stream_ids, frame_idx, cond, c0, c0_emb, codes_out, stats,
                        p.trace);
  }
  mcd_status s = launch_begin(c, n_streams, stream_ids, frame_idx, cond, c0, c0_emb);
  if (s != MCD_OK) return s;
  FrameParams p = c->fp;
  p.codes_out = codes_out;
  p.stats = stats;
  p.single_call = 0;
  p.logits_out = nullptr;
  p.emitted_out = nullptr;
  p.n_emitted_out = nullptr;
  MCD_CHECK(launch_frame_kernel(p, c->stream));
  return MCD_OK;
}

mcd_status mcd_decode_frame(mcd_ctx* c, uint32_t stream_id, uint32_t frame_idx, const float* cond,
                            const int32_t* c0, const float* c0_emb, int32_t* codes_out, mcd_frame_stats* stats) {
  return mcd_decode_frames(c, 1, &stream_id, &frame_idx, cond, c0, c0_emb, codes_out, stats);
}

mcd_status mcd_decode_frame_host(mcd_ctx* c, uint32_t stream_id, uint32_t frame_idx, const float* cond,
                                 const int32_t* c0, const float* c0_emb, int32_t* codes_out, mcd_frame_stats* stats) {
  if (!c || !codes_out || !cond) return MCD_ERR_INVALID_ARG;
  if (!c->weights_loaded) return MCD_ERR_STATE;
  const FrameParams& p = c->fp;
  if (p.C0V > 0 && !c0) return MCD_ERR_INVALID_ARG;
  if (p.C0V == 0 && !c0_emb) return MCD_ERR_INVALID_ARG;
  uint8_t* st = c->host_stage;
  uint8_t* hp = c->host_pin;
  std::memcpy(hp + stage_cond(p), cond, (size_t)p.H * 4);
  size_t in_bytes;
  if (p.C0V > 0) {
    std::memcpy(hp + stage_c0(p), c0, 4);
    in_bytes = stage_emb(p);
  } else {
    std::memcpy(hp + stage_emb(p), c0_emb, (size_t)p.H * 4);
    in_bytes = stage_codes(p);
  }
  MCD_CHECK(cudaMemcpyAsync(st, hp, in_bytes, cudaMemcpyHostToDevice, c->stream));
  float* d_cond = reinterpret_cast<float*>(st + stage_cond(p));
  float* d_emb = reinterpret_cast<float*>(st + stage_emb(p));
  int32_t* d_c0 = reinterpret_cast<int32_t*>(st + stage_c0(p));
  int32_t* d_codes = reinterpret_cast<int32_t*>(st + stage_codes(p));
  mcd_frame_stats* d_stats = reinterpret_cast<mcd_frame_stats*>(st + stage_stats(p));
  mcd_status s = mcd_decode_frame(c, stream_id, frame_idx, d_cond, p.C0V > 0 ? d_c0 : nullptr,
                                  p.C0V > 0 ? nullptr : d_emb, d_codes, d_stats);
  if (s != MCD_OK) return s;
  // codes | stats | err in one copy; the wait on the stream is the only synchronisation.
  MCD_CHECK(cudaMemcpyAsync(hp + stage_codes(p), d_codes, host_stage_bytes(p) - stage_codes(p),
                            cudaMemcpyDeviceToHost, c->stream));
  MCD_CHECK(cudaStreamSynchronize(c->stream));
  int err;
  std::memcpy(&err, hp + stage_err(p), sizeof(int));
  if (err != 0) {
    MCD_CHECK(cudaMemsetAsync(c->fp.err, 0, sizeof(int), c->stream));
    MCD_CHECK(cudaStreamSynchronize(c->stream));
    return (mcd_status)err;
  }
  std::memcpy(codes_out, hp + stage_codes(p), (size_t)p.P * 4);
  if (stats) std::memcpy(stats, hp + stage_stats(p), sizeof(mcd_frame_stats));
  return MCD_OK;
}

mcd_status mcd_set_tree(mcd_ctx* c, int32_t n_nodes, const int32_t* parent, const int32_t* rank) {
  if (!c) return MCD_ERR_INVALID_ARG;
  FrameParams& p = c->fp;
  if (p.draft_mode != MCD_DRAFT_TREE) return MCD_ERR_STATE;
  if (n_nodes < 1 || n_nodes > kMaxTree || !parent || !rank) return MCD_ERR_INVALID_ARG;
  int depth[kMaxTree], m[kMaxDraft] = {0}, maxd = 0;
  for (int i = 0; i < n_nodes; ++i) {
    if (parent[i] < -1 || parent[i] >= i || rank[i] < 0 || rank[i] >= kMaxTreeRank) return MCD_ERR_INVALID_ARG;
    depth[i] = parent[i] < 0 ? 1 : depth[parent[i]] + 1;
    if (depth[i] > p.K || rank[i] >= p.top_k) return MCD_ERR_INVALID_ARG;
    if (i > 0 && depth[i] < depth[i - 1]) return MCD_ERR_INVALID_ARG;       // breadth-first order
    for (int j = 0; j < i; ++j)
      if (parent[j] == parent[i] && rank[j] == rank[i]) return MCD_ERR_INVALID_ARG;
    m[depth[i] - 1] = std::max(m[depth[i] - 1], rank[i] + 1);
    maxd = std::max(maxd, depth[i]);
  }
  p.tree_n = n_nodes;
  p.tree_maxd = maxd;
  for (int i = 0; i < n_nodes; ++i) {
    p.tree_parent[i] = (signed char)parent[i];
    p.tree_rank[i] = (signed char)rank[i];
    p.tree_depth[i] = (signed char)depth[i];
    p.tree_anc[i] = (parent[i] < 0 ? 0ull : p.tree_anc[parent[i]]) | (1ull << i);
  }
  for (int d = 0; d < kMaxDraft; ++d) p.tree_m[d] = m[d];
  return MCD_OK;
}

mcd_status mcd_begin_frame(mcd_ctx* c, uint32_t stream_id, uint32_t frame_idx, const float* cond, const int32_t* c0,
                           const float* c0_emb) {
  if (!c) return MCD_ERR_INVALID_ARG;
  if (c->fp.draft_mode == MCD_DRAFT_TREE) return MCD_ERR_UNSUPPORTED;   // stepwise calls are chain-only
  return launch_begin(c, 1, &stream_id, &frame_idx, cond, c0, c0_emb);
}

mcd_status mcd_verify_accept(mcd_ctx* c, int32_t* emitted, int32_t* n_emitted, float* logits_out) {
  if (!c || !emitted || !n_emitted) return MCD_ERR_INVALID_ARG;
  if (!c->weights_loaded || !c->frame_begun) return MCD_ERR_STATE;
  FrameParams p = c->fp;
  p.codes_out = nullptr;
  p.stats = nullptr;
  p.single_call = 1;
  p.emitted_out = emitted;
  p.n_emitted_out = n_emitted;
  p.logits_out = logits_out;
  reset_call_counters_kernel<<<1, 64, 0, c->stream>>>(p.st, p.ctr, p.ctr_stride);
  zero_emitted_kernel<<<1, 32, 0, c->stream>>>(p.st, n_emitted);
  MCD_CHECK(cudaGetLastError());
  MCD_CHECK(launch_frame_kernel(p, c->stream));
  return MCD_OK;
}

mcd_status mcd_draft(mcd_ctx* c, int32_t pos_k, int32_t call_idx, const float* h_k, int32_t* draft_ids,
                     int32_t* q_ids, uint32_t* q_weights, float* z_out) {
  if (!c || !h_k || !draft_ids) return MCD_ERR_INVALID_ARG;
  if (!c->weights_loaded || !c->frame_begun) return MCD_ERR_STATE;
  FrameParams& p = c->fp;
  if (pos_k < 1 || pos_k >= p.P || call_idx < 0 || call_idx >= kMaxCalls) return MCD_ERR_INVALID_ARG;
  const int n_j = std::min(p.K, p.P - pos_k);
  if (n_j <= 0) return MCD_OK;
  float* z = z_out ? z_out : p.logits;  // scratch: the context's logits buffer
  const int warps = n_j * p.V;
  draft_logits_kernel<<<(warps * 32 + 255) / 256, 256, 0, c->stream>>>(p, pos_k, n_j, h_k, z);
  draft_sample_kernel<<<n_j, kConsumerThreads, sizeof(TopkScratch), c->stream>>>(p, pos_k, call_idx, z, p.topk,
                                                                                  draft_ids, q_ids, q_weights);
  MCD_CHECK(cudaGetLastError());
  return MCD_OK;
}

mcd_status mcd_accept_from_logits(mcd_ctx* c, int32_t a, int32_t n_drafts, int32_t call_idx, const float* p_logits,
                                  const float* q_logits, const int32_t* draft_ids, int32_t* emitted, int32_t* out2) {
  if (!c || !p_logits || !emitted || !out2) return MCD_ERR_INVALID_ARG;
  FrameParams& p = c->fp;
  if (!c->frame_begun) return MCD_ERR_STATE;
  if (n_drafts < 0 || n_drafts > p.K || a < 0 || a + n_drafts > p.P || a >= p.P) return MCD_ERR_INVALID_ARG;
  if (n_drafts > 0 && (!q_logits || !draft_ids)) return MCD_ERR_INVALID_ARG;
  if (call_idx < 0 || call_idx >= kMaxCalls) return MCD_ERR_INVALID_ARG;
  accept_logits_kernel<<<1, kConsumerThreads, sizeof(TopkScratch), c->stream>>>(
      p, a, n_drafts, call_idx, p_logits, q_logits, draft_ids, p.topk, emitted, out2);
  MCD_CHECK(cudaGetLastError());
  return MCD_OK;
}

mcd_status mcd_topk_softmax(mcd_ctx* c, int32_t n_rows, const float* logits, int32_t* ids, uint32_t* weights,
                            uint64_t* sums) {
  if (!c || !logits || n_rows < 0) return MCD_ERR_INVALID_ARG;
  if (n_rows == 0) return MCD_OK;
  FrameParams& p = c->fp;
  if (n_rows > 128) return MCD_ERR_UNSUPPORTED;   // the documented limit
  topk_rows_kernel<<<n_rows, kConsumerThreads, sizeof(TopkScratch), c->stream>>>(
      logits, p.V, p.top_k, p.T, p.topk, ids, weights, reinterpret_cast<unsigned long long*>(sums));
  MCD_CHECK(cudaGetLastError());
  return MCD_OK;
}

int64_t mcd_trace_bytes(const mcd_ctx* c) {
  if (!c) return 0;
  return c->fp.trace_stride * c->cfg.max_streams;
}

mcd_status mcd_set_trace(mcd_ctx* c, void* trace) {
  if (!c) return MCD_ERR_INVALID_ARG;
  c->fp.trace = static_cast<uint8_t*>(trace);
  return MCD_OK;
}

mcd_status mcd_set_timeline(mcd_ctx* c, uint64_t* timeline) {
  if (!c) return MCD_ERR_INVALID_ARG;
  c->fp.timeline = reinterpret_cast<unsigned long long*>(timeline);
  return MCD_OK;
}

}  // extern "C"

namespace {
// One thread waits with the library's bounded waits on a counter nobody increments (kind 0)
// or an mbarrier nobody arrives on (kind 1); the elapsed %globaltimer time goes to waited.
__global__ void bounded_wait_test_kernel(const unsigned* never, int* err, unsigned long long wait_ns, int kind,
                                         unsigned long long* waited) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  fence_barrier_init();
  const uint64_t t0 = globaltimer();
  bool ok;
  if (kind == 0)
    ok = wait_counter(never, 1u, err, wait_ns);
  else
    ok = wait_mbar(&bar, 0u, err, wait_ns, nullptr);
  *waited = globaltimer() - t0;
  if (ok) atomicCAS(err, 0, (int)MCD_ERR_STATE);     // cannot happen: nothing signals
}
}  // namespace

extern "C" {

mcd_status mcd_test_bounded_wait(mcd_ctx* c, int32_t kind, uint64_t wait_ns, uint64_t* waited_ns) {
  if (!c || (kind != 0 && kind != 1) || wait_ns < 1000ull || wait_ns > 10000000000ull) return MCD_ERR_INVALID_ARG;
  const FrameParams& p = c->fp;
  int pending = 0;
  MCD_CHECK(cudaStreamSynchronize(c->stream));
  MCD_CHECK(cudaMemcpy(&pending, p.err, sizeof(int), cudaMemcpyDeviceToHost));
  if (pending != 0) return MCD_ERR_STATE;
  // the 16-byte error slot of the staging area: err | never-set counter | waited (ns)
  uint8_t* slot = c->host_stage + stage_err(p);
  unsigned* never = reinterpret_cast<unsigned*>(slot + 4);
  unsigned long long* waited = reinterpret_cast<unsigned long long*>(slot + 8);
  MCD_CHECK(cudaMemsetAsync(slot + 4, 0, 12, c->stream));
  bounded_wait_test_kernel<<<1, 32, 0, c->stream>>>(never, p.err, (unsigned long long)wait_ns, kind, waited);
  MCD_CHECK(cudaGetLastError());
  MCD_CHECK(cudaStreamSynchronize(c->stream));
  unsigned long long w = 0;
  MCD_CHECK(cudaMemcpy(&w, waited, sizeof(w), cudaMemcpyDeviceToHost));
  if (waited_ns) *waited_ns = w;
  return mcd_sync(c);
}

mcd_status mcd_sync(mcd_ctx* c) {
  if (!c) return MCD_ERR_INVALID_ARG;
  MCD_CHECK(cudaStreamSynchronize(c->stream));
  int err = 0;
  MCD_CHECK(cudaMemcpy(&err, c->fp.err, sizeof(int), cudaMemcpyDeviceToHost));
  if (err != 0) {
    MCD_CHECK(cudaMemset(c->fp.err, 0, sizeof(int)));
    return (mcd_status)err;
  }
  return MCD_OK;
}

}  // extern "C"
