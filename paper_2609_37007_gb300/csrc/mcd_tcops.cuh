// The transformer-block products of many rows on the tcgen05 GEMM (mcd_tcgemm.cuh), shared by
// the batched path (many streams per call) and the CodeDecoder prompt prefill: with bf16
// weights and qkv_dim, F, H multiples of 128 the QKV, Wo, gate/up and down products run on
// the tensor cores.  Their operand rows are written as SW128 tiles by the kernel that
// produces them: the normalised rows by the pass that also folds the k-split partial sums of
// the previous residual product into the residual stream (tc_resid_norm_kernel), the
// attention outputs by the attention kernel, the SwiGLU outputs by the gate/up epilogue.
// Every kernel reads its live row count from device memory (*nrows, rows beyond it are
// neither computed nor written).  Internal linkage: each translation unit has its copy.
#pragma once
#include "mcd_internal.cuh"
#include "mcd_tcgemm.cuh"

namespace mcd {
namespace {


// Normalised operand rows x * gain / rms(x) of the call's packed rows as SW128 tiles (hi; with
// lo also the bf16 remainder), one 8-element chunk per thread.
__global__ void __launch_bounds__(256) tc_norm_operand_kernel(const float* __restrict__ X, const float* __restrict__ gain,
                                                              const float* __restrict__ ss, int H, float eps,
                                                              const int* nrows, int Rtc, uint8_t* hi, uint8_t* lo) {
  const int M = *nrows, cpr = H / 8;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < M * cpr; i += gridDim.x * blockDim.x) {
    const int r = i / cpr, ch = i - r * cpr, k = ch * 8;
    const float s = rsqrtf(ss[r] / (float)H + eps);
    const float4 x0 = __ldcg(reinterpret_cast<const float4*>(X + (size_t)r * H + k));
    const float4 x1 = __ldcg(reinterpret_cast<const float4*>(X + (size_t)r * H + k + 4));
    const float4 g0 = __ldg(reinterpret_cast<const float4*>(gain + k));
    const float4 g1 = __ldg(reinterpret_cast<const float4*>(gain + k + 4));
    const float v[8] = {x0.x * g0.x * s, x0.y * g0.y * s, x0.z * g0.z * s, x0.w * g0.w * s,
                        x1.x * g1.x * s, x1.y * g1.y * s, x1.z * g1.z * s, x1.w * g1.w * s};
    uint32_t h[4], l[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      h[q] = pack_bf16x2(v[2 * q], v[2 * q + 1]);
      l[q] = pack_bf16x2(v[2 * q] - bf16_lo_f32(h[q]), v[2 * q + 1] - bf16_hi_f32(h[q]));
    }
    const size_t off = tc::sw128_offset(Rtc, r, ch >> 3, ch & 7);
    *reinterpret_cast<uint4*>(hi + off) = make_uint4(h[0], h[1], h[2], h[3]);
    if (lo) *reinterpret_cast<uint4*>(lo + off) = make_uint4(l[0], l[1], l[2], l[3]);
  }
}

// Row-major bf16 [rows][K] -> an SW128-tiled matrix of R rows (weight load): source row r
// goes to row row0 + (r / grp) * gstride + r % grp (grp = rows: row0 + r).
__global__ void tc_weight_tile_kernel(const uint16_t* __restrict__ src, int rows, int K, int R, int row0, int grp,
                                      int gstride, uint8_t* __restrict__ dst) {
  const long long total = (long long)rows * (K / 8);
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < total; i += (long long)gridDim.x * blockDim.x) {
    const int r = (int)(i / (K / 8)), ch = (int)(i % (K / 8));
    const int dr = row0 + (r / grp) * gstride + r % grp;
    *reinterpret_cast<uint4*>(dst + tc::sw128_offset(R, dr, ch >> 3, ch & 7)) =
        *reinterpret_cast<const uint4*>(src + (size_t)r * K + (size_t)ch * 8);
  }
}

constexpr int kTcBN = 128;        // packed rows per tile: QKV (hi + lo operand), Wo, down
constexpr int kTcSplit = 6;       // k-splits of the residual products (at most)
// Splits of the residual products at Rtc packed rows: four (128-column tiles, 128 CTAs at 512
// rows) from 512 rows on, where more splits' partial sums cost more than they save; six below
// (3 x 8 x 6 = 144 CTAs at 128 rows, where 128-column tiles would leave 32 CTAs).
inline int tc_resid_split(int Rtc) { return Rtc >= 512 ? 4 : kTcSplit; }

// q, k, v = W (x . g / rms) with the hi + lo operand.
__global__ void __launch_bounds__(tc::kPThreads, 1) tc_qkv_kernel(const tc::GemmArgs g, float* out, int ld,
                                                                   const int* nrows) {
  const int M = *nrows;
  tc::gemm_persistent<kTcBN, false, true>(g, 1, [&](int m, int n, int, float v, float) {
    if (n < M) out[(size_t)n * ld + m] = v;
  });
}

// gate/up -> SwiGLU, one 128 x pitch tile per CTA (gemm_tile_run).  A is the interleaved
// gate/up matrix of 2F rows written by tc_tile_layer: rows 0..63 of tile b are the gate rows
// of features 64b..64b+63, rows 64..127 the up rows of the same features.  The accumulator is
// staged in shared memory (the idle operand ring, [column][tile row]) so that a thread holds
// the gate and up values of eight consecutive features of one packed row; it writes
// silu(gate) * up as one 16-byte bf16 chunk of the down product's SW128 operand (k-slice b,
// element (row n, feature m)).  Packed rows at or past *nrows are not written.
constexpr int kGuThreads = 256;
template <int BN>
__global__ void __launch_bounds__(kGuThreads, 1) tc_gu_kernel(const tc::GemmArgs g, uint8_t* act_t, int Rtc,
                                                               const int* nrows) {
  using L = tc::Layout<BN>;
  constexpr int kSP = tc::kBM + 4;                  // staged column stride (floats)
  static_assert((size_t)BN * kSP * 4 <= (size_t)L::kStages * L::kStageBytes, "gate/up staging exceeds the ring");
  tc::TileRun t;
  if (!tc::gemm_tile_run<BN, false, false>(g, t)) return;
  float* S = reinterpret_cast<float*>(t.smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int quarter = warp & 3, part = warp >> 2, n_parts = (int)(blockDim.x >> 7);
  if (t.ok) {
    // warp w drains TMEM lanes 32 (w % 4) .. (tile rows) for the column chunks c = w / 4 mod
    // (warps / 4); a warp's 32 lanes store 32 consecutive floats of one column
    const uint32_t lane_base = t.tmem + ((uint32_t)(quarter * 32) << 16);
    const int r = quarter * 32 + lane, n_ch = t.nw >> 4;
    for (int ch = part; ch < n_ch; ch += n_parts) {
      float v[16];
      tc::tmem_ld16(lane_base + (uint32_t)(16 * ch), v);
#pragma unroll
      for (int j = 0; j < 16; ++j) S[(16 * ch + j) * kSP + r] = v[j];
    }
  }
  __syncthreads();
  if (t.ok) {
    const int M = *nrows, kt = t.m0 / tc::kBM;
    for (int it = threadIdx.x; it < t.nw * 8; it += blockDim.x) {
      const int nl = it >> 3, c = it & 7, n = t.n0 + nl;
      if (n >= M) continue;
      const float4* gs = reinterpret_cast<const float4*>(S + nl * kSP + 8 * c);
      const float4* us = reinterpret_cast<const float4*>(S + nl * kSP + 64 + 8 * c);
      const float4 g0 = gs[0], g1 = gs[1], u0 = us[0], u1 = us[1];
      const float gt[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
      const float up[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
      float v[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) v[e] = gt[e] / (1.0f + __expf(-gt[e])) * up[e];
      *reinterpret_cast<uint4*>(act_t + tc::sw128_offset(Rtc, n, kt, c)) =
          make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]), pack_bf16x2(v[4], v[5]),
                     pack_bf16x2(v[6], v[7]));
    }
  }
  tc::gemm_tile_free<BN, false, false>(t);
}

// Residual products (Wo, down): one 128 x pitch tile per CTA over the k-slices of split
// blockIdx.z of kTcSplit; split z writes its partial sums part[z][n][m] (plain stores);
// tc_resid_norm_kernel adds them into the residual stream.
constexpr int kResidThreads = 256;
template <int BN>
__global__ void __launch_bounds__(kResidThreads, 1) tc_resid_kernel(const tc::GemmArgs g, float* part, int ld, int Rtc,
                                                                     const int* nrows) {
  const int M = *nrows;
  const size_t zoff = (size_t)blockIdx.z * Rtc;
  tc::gemm_tile<BN, false, false>(g, [&](int m, int n, float v, float) {
    if (n < M) part[(zoff + n) * ld + m] = v;
  });
}

// Per packed row (one CTA, thread t owns elements 8t..8t+7): X += the nz partial sums, the
// row's sum of squares (the next RMSNorm), and with a gain the next product's normalised
// operand (hi; with lo also the remainder) as SW128 tiles.
__global__ void __launch_bounds__(128) tc_resid_norm_kernel(float* X, const float* __restrict__ part, int nz, int Rtc,
                                                            int H, const int* nrows, float* ss_out,
                                                            const float* __restrict__ gain, float eps, uint8_t* hi,
                                                            uint8_t* lo) {
  const int r = blockIdx.x;
  if (r >= *nrows) return;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const bool live = t < H / 8;
  __shared__ float red[4];
  float x[8];
  float ss = 0.f;
  if (live) {
    float4* xr = reinterpret_cast<float4*>(X + (size_t)r * H + 8 * t);
    float4 a = xr[0], b = xr[1];
    // every partial's loads issued before the first add (nz <= kTcSplit), added in split order
    float4 u[kTcSplit], w[kTcSplit];
#pragma unroll
    for (int z = 0; z < kTcSplit; ++z) {
      if (z < nz) {
        const float4* pr = reinterpret_cast<const float4*>(part + ((size_t)z * Rtc + r) * H + 8 * t);
        u[z] = __ldcg(pr);
        w[z] = __ldcg(pr + 1);
      }
    }
#pragma unroll
    for (int z = 0; z < kTcSplit; ++z) {
      if (z < nz) {
        a.x += u[z].x; a.y += u[z].y; a.z += u[z].z; a.w += u[z].w;
        b.x += w[z].x; b.y += w[z].y; b.z += w[z].z; b.w += w[z].w;
      }
    }
    xr[0] = a;
    xr[1] = b;
    x[0] = a.x; x[1] = a.y; x[2] = a.z; x[3] = a.w; x[4] = b.x; x[5] = b.y; x[6] = b.z; x[7] = b.w;
#pragma unroll
    for (int i = 0; i < 8; ++i) ss += x[i] * x[i];
  }
#pragma unroll
  for (int off = 16; off; off >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, off);
  if (lane == 0) red[warp] = ss;
  __syncthreads();
  const float tot = red[0] + red[1] + red[2] + red[3];
  if (t == 0) ss_out[r] = tot;
  if (gain && live) {
    const float s = rsqrtf(tot / (float)H + eps);
    const float4 g0 = __ldg(reinterpret_cast<const float4*>(gain + 8 * t));
    const float4 g1 = __ldg(reinterpret_cast<const float4*>(gain + 8 * t + 4));
    const float v[8] = {x[0] * g0.x * s, x[1] * g0.y * s, x[2] * g0.z * s, x[3] * g0.w * s,
                        x[4] * g1.x * s, x[5] * g1.y * s, x[6] * g1.z * s, x[7] * g1.w * s};
    uint32_t h[4], l[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      h[q] = pack_bf16x2(v[2 * q], v[2 * q + 1]);
      l[q] = pack_bf16x2(v[2 * q] - bf16_lo_f32(h[q]), v[2 * q + 1] - bf16_hi_f32(h[q]));
    }
    const size_t off = tc::sw128_offset(Rtc, r, t >> 3, t & 7);
    *reinterpret_cast<uint4*>(hi + off) = make_uint4(h[0], h[1], h[2], h[3]);
    if (lo) *reinterpret_cast<uint4*>(lo + off) = make_uint4(l[0], l[1], l[2], l[3]);
  }
}

// Non-empty k-splits of a residual product over K in z splits (gemm_tile's split of the
// k-slices).
static int tc_splits(int K, int z) {
  const int nk = K / tc::kBK, per = (nk + z - 1) / z;
  return (nk + per - 1) / per;
}


// The transformer-block products can use the tensor-core GEMM (shape and dtype limits).
bool tc_block_supported(const FrameParams& p) {
  return p.wdtype == MCD_WEIGHT_BF16 && p.qkv_dim % 128 == 0 && p.F % 128 == 0 && p.H % 128 == 0 &&
         (p.NH * p.D) % 64 == 0 && p.H % 64 == 0 && p.F % 64 == 0 && p.H <= 1024;
}

// SW128 copies of one layer's weights: [qkv | gate/up interleaved (2F rows) | o | d], offsets
// within a layer.
struct TcLayerOffsets {
  size_t qkv = 0, gu = 0, o = 0, d = 0, layer = 0;
};
inline TcLayerOffsets tc_layer_offsets(const FrameParams& p) {
  TcLayerOffsets t;
  const size_t H = p.H, F = p.F, qd = (size_t)p.NH * p.D;
  t.qkv = 0;
  t.gu = t.qkv + (size_t)p.qkv_dim * H * 2;
  t.o = t.gu + 2 * F * H * 2;
  t.d = t.o + H * qd * 2;
  t.layer = t.d + H * F * 2;
  return t;
}
// Tile layer l's row-major bf16 sources (device) into the SW128 copies at base.
inline void tc_tile_layer(const FrameParams& p, cudaStream_t st, const uint8_t* wq, const uint8_t* wk, const uint8_t* wv,
                          const uint8_t* wo, const uint8_t* wg, const uint8_t* wu, const uint8_t* wd, uint8_t* base) {
  const TcLayerOffsets t = tc_layer_offsets(p);
  const int H = p.H, F = p.F, qd = p.NH * p.D, kd = p.NKV * p.D;
  auto tile = [&](const uint8_t* s, int rows, int K, int R, int row0, int grp, int gstride, size_t off) {
    tc_weight_tile_kernel<<<512, 256, 0, st>>>(reinterpret_cast<const uint16_t*>(s), rows, K, R, row0, grp, gstride,
                                               base + off);
  };
  tile(wq, qd, H, p.qkv_dim, 0, qd, 0, t.qkv);
  tile(wk, kd, H, p.qkv_dim, qd, kd, 0, t.qkv);
  tile(wv, kd, H, p.qkv_dim, qd + kd, kd, 0, t.qkv);
  // gate rows 64b.. of tile b at its rows 0..63, the up rows at 64..127 (tc_gu_kernel)
  tile(wg, F, H, 2 * F, 0, 64, 128, t.gu);
  tile(wu, F, H, 2 * F, 64, 64, 128, t.gu);
  tile(wo, H, qd, H, 0, H, 0, t.o);
  tile(wd, H, F, H, 0, F, 0, t.d);
}
// Dynamic shared memory of the block kernels (once per translation unit).
inline cudaError_t tc_block_set_smem() {
  cudaError_t e = cudaFuncSetAttribute(tc_qkv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       tc::PLayout<kTcBN, false, true>::kSmemBytes);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(tc_gu_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, tc::Layout<128>::kSmemBytes);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(tc_gu_kernel<176>, cudaFuncAttributeMaxDynamicSharedMemorySize, tc::Layout<176>::kSmemBytes);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(tc_gu_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize, tc::Layout<256>::kSmemBytes);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(tc_resid_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             tc::Layout<128>::kSmemBytes);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(tc_resid_kernel<176>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             tc::Layout<176>::kSmemBytes);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(tc_resid_kernel<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             tc::Layout<256>::kSmemBytes);
  return e;
}

// Persistent launch shape: one CTA per SM at most, one per tile at least.
inline dim3 tc_grid(int n_tiles, int n_sm) { return dim3(n_tiles < n_sm ? n_tiles : n_sm); }
inline int tc_tiles(int N, int BN, int M, int splits) { return (N / BN) * (M / tc::kBM) * splits; }

// gate/up -> SwiGLU into the down product's operand.  gu: the interleaved gate/up matrix
// (2F rows); xn: the normalised operand of Rtc rows.  The tile pitch over the packed rows fills
// the SMs with one tile per CTA (three tiles of 176 / 176 / 160 rows at 512 rows, F = 3072).
inline void tc_launch_gu(const uint8_t* gu, const uint8_t* xn, uint8_t* act_t, int Rtc, const int* nrows, int F,
                         int H, int* err, unsigned long long wait_ns, int n_sm, cudaStream_t s) {
  const int pitch = tc::tile_pitch(2 * F, Rtc, n_sm);
  const tc::GemmArgs g{gu, nullptr, xn, nullptr, 2 * F, Rtc, H, nrows, err, wait_ns, pitch};
  const dim3 grid((Rtc + pitch - 1) / pitch, 2 * F / tc::kBM);
  if (pitch <= 128)
    tc_gu_kernel<128><<<grid, kGuThreads, tc::Layout<128>::kSmemBytes, s>>>(g, act_t, Rtc, nrows);
  else if (pitch <= 176)
    tc_gu_kernel<176><<<grid, kGuThreads, tc::Layout<176>::kSmemBytes, s>>>(g, act_t, Rtc, nrows);
  else
    tc_gu_kernel<256><<<grid, kGuThreads, tc::Layout<256>::kSmemBytes, s>>>(g, act_t, Rtc, nrows);
}

// Wo or down (A = w: H rows of K, B = act: Rtc rows) -> tc_resid_split(Rtc) partial sums.
// T column tiles x (H / 128) weight tiles x z splits fill the SMs with one tile per CTA
// (H = 1024: T = 4 of 128 packed rows at 512 rows, 128 CTAs; T = 3 of 48 / 48 / 32 at 128
// rows, 144 CTAs).
inline void tc_launch_resid(const uint8_t* w, const uint8_t* act, float* part, int H, int Rtc, int K, const int* nrows,
                            int* err, unsigned long long wait_ns, int n_sm, cudaStream_t s) {
  const int n_mt = H / tc::kBM, units = Rtc / 16, z = tc_resid_split(Rtc);
  int T = n_sm / (n_mt * z);
  if (T < 1) T = 1;
  if (T < (Rtc + 255) / 256) T = (Rtc + 255) / 256;
  if (T > units) T = units;
  const int pitch = (units + T - 1) / T * 16;
  const tc::GemmArgs g{w, nullptr, act, nullptr, H, Rtc, K, nrows, err, wait_ns, pitch};
  const dim3 grid((Rtc + pitch - 1) / pitch, n_mt, z);
  if (pitch <= 128)
    tc_resid_kernel<128><<<grid, kResidThreads, tc::Layout<128>::kSmemBytes, s>>>(g, part, H, Rtc, nrows);
  else if (pitch <= 176)
    tc_resid_kernel<176><<<grid, kResidThreads, tc::Layout<176>::kSmemBytes, s>>>(g, part, H, Rtc, nrows);
  else
    tc_resid_kernel<256><<<grid, kResidThreads, tc::Layout<256>::kSmemBytes, s>>>(g, part, H, Rtc, nrows);
}

}  // namespace
}  // namespace mcd
