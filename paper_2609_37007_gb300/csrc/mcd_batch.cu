// Batched decoding of many independent streams (up to 128 streams, 512 packed rows per
// call): the per-frame draft-and-verify loop of arXiv 2609.37007 (Sec. 2.2, Fig. 3) for
// every stream at once, with the rows of all unfinished streams re-packed every call.
//
// With hundreds of rows per call the weight matrices are multiplied as real GEMMs, so this
// path is a sequence of grid-wide kernels per call instead of the persistent frame kernel:
//
//   pack -> embed -> 5 x [QKV GEMM -> attention -> Wo GEMM (+residual) -> gate/up GEMM
//   (SwiGLU) -> down GEMM (+residual)] -> LM-head GEMM (grouped by head) -> top-k -> accept
//
// captured once per context as a CUDA graph holding n_pos call bodies (a call never emits
// fewer than one code, so n_pos calls always finish a frame; bodies after the last active
// call find no rows and return at once).  RMSNorm never gets its own pass.  With bf16
// weights whose widths are multiples of 128 (the MultiCodeDecoder's) every product runs on
// the tcgen05 GEMM (mcd_tcgemm.cuh, block kernels in mcd_tcops.cuh): weights and operand
// rows as 128-byte swizzled tiles, TMEM accumulators, the residual products split over k
// into partial sums that one per-row pass folds into the residual stream while it writes
// the next product's normalised operand.  Other shapes use the mma.sync GEMM below (the
// weights in the frame kernel's tiled unit layout, 128 weight rows x 64 packed rows per CTA
// through a 4-stage cp.async pipeline, the norm folded into the operand staging).  Sampling
// and acceptance use the same integer sampler as the frame kernel.
#include <algorithm>
#include <cstring>
#include <vector>

#include "mcd_host.cuh"
#include "mcd_internal.cuh"
#include "mcd_sampler.cuh"
#include "mcd_tcgemm.cuh"
#include "mcd_tcops.cuh"

namespace mcd {

constexpr int kGM = 128;                 // weight rows per GEMM tile (8 m-tiles)
constexpr int kGN = 64;                  // packed rows per GEMM tile (8 n-tiles)
constexpr int kGK = 64;                  // k per pipeline stage (4 k-tiles)
constexpr int kGStages = 4;
constexpr int kGBStride = kGK + 8;       // bf16 per staged operand row (144 B: conflict-free ldmatrix)
constexpr int kGAStage = 32 * 512;       // 8 m-tiles x 4 k-tiles of 512 B
constexpr int kGBStage = kGN * kGBStride * 2;
constexpr int kGStagesHilo = 3;          // with the hi + lo operand: two CTAs per SM still fit
constexpr int kGemmSmem = kGStages * (kGAStage + kGBStage);
constexpr int kGemmSmemHilo = kGStagesHilo * (kGAStage + 2 * kGBStage);
constexpr int kRecSlots = kMaxDraft + 1;   // distributions per packed row (verify + drafts)
constexpr int kBatchQVec = 16;             // query vectors per attention CTA: rows x (q heads per KV head)
constexpr int kBatchKeys = 16;             // keys of a frame: positions 0..15 (c15 is never fed)

// Operand rows: fp32 rows normalised while staged (as one bf16, or as a bf16 hi + lo pair
// carrying about 16 mantissa bits, for the QKV and LM-head products whose errors the
// attention softmax and the sampler see directly), or rows already in bf16.
enum BSrc { BSRC_NORM = 0, BSRC_BF16 = 1, BSRC_NORM_HILO = 2 };
enum Epi { EPI_QKV = 0, EPI_RESID = 1, EPI_SWIGLU = 2, EPI_HEADS = 3 };

struct BatchRow {
  int s, n, pos, id;
  const uint8_t* src;     // layer-0 input row
  int f32;                // src is fp32 (else bf16)
};

struct BatchInfo {
  int M;                  // packed rows of the call
  int n_pairs;            // (row, j) distributions of the call
  int head_rows[16];      // rows reading LM head P (entries in head_list)
  int head_off[16];
};

// Per-frame arguments, copied to the device before each graph launch.
struct BatchFrame {
  int S;
  unsigned stream_ids[kMaxBatchStreams];
  unsigned frame_ids[kMaxBatchStreams];
  const float* cond;
  const int* c0;
  const float* c0emb;
  int* codes_out;
  mcd_frame_stats* stats;
  uint8_t* trace;
};

struct BatchBufs {
  int R;                  // packed-row capacity
  BatchInfo* info;
  BatchFrame* frame;
  BatchRow* rows;         // [R]
  int* sbase;             // [kMaxBatchStreams] first packed row of each stream (-1: inactive)
  int* pairs;             // [R * kRecSlots] (row << 3) | j
  int* head_list;         // [R * kRecSlots] grouped by head
  float* X;               // [R][H] residual stream
  float* ss;              // [2L + 1][R] per-row sums of squares of X after each residual write
  float* qkv;             // [R][qkv_dim]
  uint16_t* att;          // [R][NH * D] bf16 attention outputs
  uint16_t* act;          // [R][F] bf16 SwiGLU outputs
  float* logits;          // [R][kRecSlots][V]
  TopkRec* recs;          // [2][R][kRecSlots]
  // tensor-core GEMM operands (SW128 tiles of Rtc rows, Rtc = R rounded up to 128)
  int Rtc;
  uint8_t* xn_hi;         // normalised rows, bf16 (and the low halves for the QKV product)
  uint8_t* xn_lo;
  uint8_t* att_t;         // attention outputs
  uint8_t* act_t;         // SwiGLU outputs
  float* part;            // [kTcSplit][Rtc][H] k-split partial sums of the residual products
  int Qcap;               // LM-head operand rows: every (row, j) pair, groups padded per head
  uint8_t* hq_hi;         // LM-head operand (normalised rows of the pairs, grouped by head)
  uint8_t* hq_lo;
};

// Weights of the tensor-core GEMMs: per layer the row-major matrices as SW128 tiles.
struct TcWeights {
  uint8_t* arena = nullptr;
  TcLayerOffsets off;                                         // within a layer, layer stride
  uint8_t* heads = nullptr;                                   // [n_pos][V x H] SW128 tiles
};

// ------------------------------------------------------------------------------------
// small helpers
// ------------------------------------------------------------------------------------
__device__ __forceinline__ void cp_async16(void* dst, const void* src, int src_bytes) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(dst)), "l"(src), "r"(src_bytes)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}
__device__ __forceinline__ uint16_t f32_to_bf16(float x) { return (uint16_t)bf16_rn_bits(x); }

// Offset (bytes) of 16 x 16 tile (m-tile mt, k-tile kt) in a tiled bf16 matrix.
__device__ __forceinline__ size_t tile_byte_offset(const MatGeom& g, int mt, int kt) {
  const int kcu = kt / g.Ku, ktl = kt - kcu * g.Ku, mbu = mt / g.Mu, mi = mt - mbu * g.Mu;
  const long long u = (long long)kcu * g.n_mb + mbu;
  return (size_t)(((u * g.Mu + mi) * g.Ku) + ktl) * 512;
}

// ------------------------------------------------------------------------------------
// pack: the call's rows, distributions and head groups from every stream's state
// ------------------------------------------------------------------------------------
__global__ void __launch_bounds__(256) batch_pack_kernel(FrameParams p, BatchBufs b) {
  __shared__ int s_cnt[256], s_pc[256], s_head[16], s_hcur[16];
  const BatchFrame* fa = b.frame;
  const int S = fa->S, tid = threadIdx.x;
  const int L = p.L;
  for (int i = tid; i < (2 * L + 1) * b.R; i += blockDim.x) b.ss[i] = 0.f;
  if (tid < 16) s_head[tid] = 0;
  int nr = 0, np = 0;
  DevState st;
  if (tid < S) {
    st = p.st[tid];
    if (!st.done) {
      nr = st.n_rows;
      for (int n = 0; n < nr; ++n) {
        const int pos = st.pos0 + n;
        if (pos >= 1) np += min(p.K, p.P - pos) + 1;
      }
    }
  }
  // inclusive scans of (rows, pairs) over the streams: within each warp by shuffles, then
  // over the 8 warp totals
  const int lane = tid & 31, warp = tid >> 5;
  int cr = nr, cp = np;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int a = __shfl_up_sync(0xFFFFFFFFu, cr, off), c = __shfl_up_sync(0xFFFFFFFFu, cp, off);
    if (lane >= off) {
      cr += a;
      cp += c;
    }
  }
  if (lane == 31) {
    s_cnt[warp] = cr;
    s_pc[warp] = cp;
  }
  __syncthreads();
  if (warp == 0) {
    int wr = lane < 8 ? s_cnt[lane] : 0, wp = lane < 8 ? s_pc[lane] : 0;
#pragma unroll
    for (int off = 1; off < 8; off <<= 1) {
      const int a = __shfl_up_sync(0xFFFFFFFFu, wr, off), c = __shfl_up_sync(0xFFFFFFFFu, wp, off);
      if (lane >= off) {
        wr += a;
        wp += c;
      }
    }
    if (lane < 8) {
      s_cnt[8 + lane] = wr;             // inclusive totals through warp `lane`
      s_pc[8 + lane] = wp;
    }
  }
  __syncthreads();
  if (warp > 0) {
    cr += s_cnt[8 + warp - 1];
    cp += s_pc[8 + warp - 1];
  }
  const int base = cr - nr, pbase = cp - np;
  if (tid < S && nr > 0) {
    for (int n = 0; n < nr; ++n) {
      const int pos = st.pos0 + n, r = base + n;
      int id = st.pos0 == 0 ? (n == 0 ? -1 : st.codes[0]) : (n == 0 ? st.codes[st.a] : st.drafts[n - 1]);
      BatchRow row;
      row.s = tid;
      row.n = n;
      row.pos = pos;
      if (pos == 0 || (pos == 1 && p.C0V == 0)) {
        row.src = reinterpret_cast<const uint8_t*>((pos == 0 ? fa->cond : fa->c0emb) + (size_t)tid * p.H);
        row.f32 = 1;
      } else {
        const int table = pos - 1;
        if (id < 0 || id >= (table == 0 ? p.C0V : p.V)) {
          atomicCAS(p.err, 0, (int)MCD_ERR_INVALID_ARG);
          id = 0;
        }
        row.src = p.embed + (long long)table * p.embed_stride + (long long)id * p.H * 2;
        row.f32 = 0;
      }
      row.id = id;
      b.rows[r] = row;
      if (pos >= 1) {
        const int kn = min(p.K, p.P - pos);
        for (int j = 0; j <= kn; ++j) atomicAdd(&s_head[pos + j], 1);
      }
    }
  }
  if (tid < kMaxBatchStreams) b.sbase[tid] = (tid < S && nr > 0) ? base : -1;
  __syncthreads();
  if (tid == 0) {
    int off = 0;
    for (int P = 0; P < 16; ++P) {
      b.info->head_rows[P] = s_head[P];
      b.info->head_off[P] = off;
      s_hcur[P] = off;
      off += s_head[P];
    }
    b.info->M = s_cnt[8 + 7];
    b.info->n_pairs = s_pc[8 + 7];
  }
  __syncthreads();
  if (tid < S && nr > 0) {
    int pi = pbase;
    for (int n = 0; n < nr; ++n) {
      const int pos = st.pos0 + n, r = base + n;
      if (pos < 1) continue;
      const int kn = min(p.K, p.P - pos);
      for (int j = 0; j <= kn; ++j) {
        b.pairs[pi++] = (r << 3) | j;
        b.head_list[atomicAdd(&s_hcur[pos + j], 1)] = (r << 3) | j;
      }
    }
  }
}

// embed: X[r] = the row's input vector; ss[0][r] = sum of squares.
__global__ void __launch_bounds__(256) batch_embed_kernel(FrameParams p, BatchBufs b) {
  const int r = blockIdx.x;
  if (r >= b.info->M) return;
  const BatchRow row = b.rows[r];
  float s = 0.f;
  for (int k = threadIdx.x; k < p.H; k += blockDim.x) {
    const float v = row.f32 ? __ldg(reinterpret_cast<const float*>(row.src) + k)
                            : bf16_bits_to_f32(__ldg(reinterpret_cast<const uint16_t*>(row.src) + k));
    b.X[(size_t)r * p.H + k] = v;
    s += v * v;
  }
  for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
  __shared__ float sw[8];
  if ((threadIdx.x & 31) == 0) sw[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) t += sw[w];
    b.ss[r] = t;
  }
}

// ------------------------------------------------------------------------------------
// GEMM: C[o][row] = sum_k W[o][k] X[row][k] over 128 weight rows x 64 packed rows per CTA
// ------------------------------------------------------------------------------------
struct GemmArgs {
  const uint8_t* W;       // tiled bf16 matrix (heads: head 1; head P at + (P-1) * g.stride)
  MatGeom g;
  // operand rows
  const float* X;         // BSRC_NORM: fp32 rows [R][ldx], scaled by gain[k] / rms(row)
  const float* gain;
  const float* ss;        // per-row sums of squares of X
  const uint16_t* Xb;     // BSRC_BF16: bf16 rows [R][ldx]
  int ldx;
  // outputs
  float* out;             // EPI_QKV: [R][ld]; EPI_RESID: the residual X [R][ld]
  uint16_t* act;          // EPI_SWIGLU: [R][ld]
  int ld;
  float* logits;          // EPI_HEADS: [R][kRecSlots][V]
  const float* head_bias; // EPI_HEADS: [n_pos][K][V]
  int K, V;
  const BatchInfo* info;
  const int* head_list;
  float eps;
};

template <int BSRC, int EPI>
__global__ void __launch_bounds__(256) batch_gemm_kernel(const __grid_constant__ GemmArgs a) {
  constexpr bool kNorm = BSRC != BSRC_BF16, kHilo = BSRC == BSRC_NORM_HILO;
  constexpr int kStages = kHilo ? kGStagesHilo : kGStages;
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ int s_row[kGN];
  __shared__ int s_j[kGN];
  __shared__ float s_inv[kGN];
  __shared__ float s_ss[kGN];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const BatchInfo* info = a.info;
  int n_rows;
  const int* rlist = nullptr;
  const uint8_t* W = a.W;
  int P = 0;
  if (EPI == EPI_HEADS) {
    P = blockIdx.z + 1;
    n_rows = info->head_rows[P];
    rlist = a.head_list + info->head_off[P];
    W += (size_t)(P - 1) * a.g.stride;
  } else {
    n_rows = info->M;
  }
  const int r0 = blockIdx.y * kGN;
  if (r0 >= n_rows) return;
  const MatGeom& g = a.g;
  const int mt0 = blockIdx.x * (kGM / 16);                 // first m-tile of the CTA
  const int n_mt = g.M >> 4;
  const int Kdim = g.K;
  // k-chunks of this CTA: all of them, or (residual GEMMs) slice blockIdx.z of gridDim.z
  int kc0 = 0, kc1 = Kdim / kGK;
  if (EPI != EPI_HEADS && gridDim.z > 1) {
    const int per = (kc1 + gridDim.z - 1) / gridDim.z;
    kc0 = blockIdx.z * per;
    kc1 = min(kc1, kc0 + per);
    if (kc0 >= kc1) return;
  }
  const int n_kc = kc1 - kc0;
  if (tid < kGN) {
    const int i = r0 + tid;
    int r = -1, j = 0;
    if (i < n_rows) {
      if (rlist) {
        const int e = rlist[i];
        r = e >> 3;
        j = e & 7;
      } else {
        r = i;
      }
    }
    s_row[tid] = r;
    s_j[tid] = j;
    if (kNorm) s_inv[tid] = r >= 0 ? rsqrtf(a.ss[r] / (float)Kdim + a.eps) : 0.f;
    s_ss[tid] = 0.f;
  }
  __syncthreads();
  uint8_t* sA = smem;
  uint16_t* sB = reinterpret_cast<uint16_t*>(smem + kStages * kGAStage);
  uint16_t* sBl = sB + (size_t)kStages * kGN * kGBStride;   // lo parts (hi/lo operand)

  // ---- stage loaders ------------------------------------------------------------------------
  auto load_A = [&](int kc, int st) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int c = tid + 256 * i, t = c >> 5, part = c & 31;
      const int mt = mt0 + (t >> 2), kt = kc * 4 + (t & 3);
      uint8_t* dst = sA + st * kGAStage + t * 512 + part * 16;
      const bool ok = mt < n_mt;
      const uint8_t* src = W + (ok ? tile_byte_offset(g, mt, kt) : 0) + part * 16;
      cp_async16(dst, src, ok ? 16 : 0);
    }
  };
  float4 breg[4];
  auto fetch_B = [&](int kc) {           // BSRC_NORM: fp32 rows into registers
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int c = tid + 256 * i, rr = c >> 4, q = c & 15;
      const int r = s_row[rr];
      breg[i] = r >= 0 ? __ldcg(reinterpret_cast<const float4*>(a.X + (size_t)r * a.ldx + kc * kGK) + q)
                       : make_float4(0.f, 0.f, 0.f, 0.f);
    }
  };
  auto store_B = [&](int kc, int st) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int c = tid + 256 * i, rr = c >> 4, q = c & 15, k = kc * kGK + 4 * q;
      const float4 gg = __ldg(reinterpret_cast<const float4*>(a.gain + k));
      const float s = s_inv[rr];
      const float x0 = breg[i].x * gg.x * s, x1 = breg[i].y * gg.y * s, x2 = breg[i].z * gg.z * s,
                  x3 = breg[i].w * gg.w * s;
      const uint32_t h01 = pack_bf16x2(x0, x1), h23 = pack_bf16x2(x2, x3);
      const size_t off = (size_t)st * (kGN * kGBStride) + rr * kGBStride + 4 * q;
      *reinterpret_cast<uint2*>(sB + off) = make_uint2(h01, h23);
      if (kHilo) {
        const uint32_t l01 = pack_bf16x2(x0 - bf16_lo_f32(h01), x1 - bf16_hi_f32(h01));
        const uint32_t l23 = pack_bf16x2(x2 - bf16_lo_f32(h23), x3 - bf16_hi_f32(h23));
        *reinterpret_cast<uint2*>(sBl + off) = make_uint2(l01, l23);
      }
    }
  };
  auto load_B16 = [&](int kc, int st) {   // BSRC_BF16: cp.async
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int c = tid + 256 * i, rr = c >> 3, ch = c & 7;
      const int r = s_row[rr];
      const uint16_t* src = a.Xb + (size_t)(r >= 0 ? r : 0) * a.ldx + kc * kGK + ch * 8;
      cp_async16(sB + (size_t)st * (kGN * kGBStride) + rr * kGBStride + ch * 8, src, r >= 0 ? 16 : 0);
    }
  };

  // ---- main loop ------------------------------------------------------------------------------
  const int wm = (warp & 3) * 2;          // the warp's first m-tile within the CTA tile
  const int wn = (warp >> 2) * 4;         // its first n-tile
  float acc[2][4][4];
#pragma unroll
  for (int i = 0; i < 2; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j)
#pragma unroll
      for (int e = 0; e < 4; ++e) acc[i][j][e] = 0.f;

#pragma unroll
  for (int st = 0; st < kStages - 1; ++st) {
    if (st < n_kc) {
      load_A(kc0 + st, st);
      if (!kNorm) {
        load_B16(kc0 + st, st);
      } else {
        fetch_B(kc0 + st);
        store_B(kc0 + st, st);
      }
    }
    cp_async_commit();
  }
  for (int it = 0; it < n_kc; ++it) {
    const int st = it % kStages;
    const int nk = it + kStages - 1;
    if (kNorm && nk < n_kc) fetch_B(kc0 + nk);
    cp_async_wait<kStages - 2>();
    __syncthreads();
    const uint8_t* A = sA + st * kGAStage;
    const uint16_t* B = sB + (size_t)st * (kGN * kGBStride);
    const uint16_t* Bl = sBl + (size_t)st * (kGN * kGBStride);
#pragma unroll
    for (int kt = 0; kt < 4; ++kt) {
      const uint4 a0 = *reinterpret_cast<const uint4*>(A + ((wm + 0) * 4 + kt) * 512 + lane * 16);
      const uint4 a1 = *reinterpret_cast<const uint4*>(A + ((wm + 1) * 4 + kt) * 512 + lane * 16);
#pragma unroll
      for (int hp = 0; hp < 2; ++hp) {
        uint32_t bf[4];
        const int row = (wn + 2 * hp + (lane >> 4)) * 8 + (lane & 7);
        const int kk = kt * 16 + ((lane >> 3) & 1) * 8;
        ldmatrix_x4(bf, B + row * kGBStride + kk);
        mma_bf16_16816(acc[0][2 * hp], a0, bf[0], bf[1]);
        mma_bf16_16816(acc[0][2 * hp + 1], a0, bf[2], bf[3]);
        mma_bf16_16816(acc[1][2 * hp], a1, bf[0], bf[1]);
        mma_bf16_16816(acc[1][2 * hp + 1], a1, bf[2], bf[3]);
        if (kHilo) {
          ldmatrix_x4(bf, Bl + row * kGBStride + kk);
          mma_bf16_16816(acc[0][2 * hp], a0, bf[0], bf[1]);
          mma_bf16_16816(acc[0][2 * hp + 1], a0, bf[2], bf[3]);
          mma_bf16_16816(acc[1][2 * hp], a1, bf[0], bf[1]);
          mma_bf16_16816(acc[1][2 * hp + 1], a1, bf[2], bf[3]);
        }
      }
    }
    // stage nk % kStages was last read in iteration it - 1, which every warp has left
    if (nk < n_kc) {
      const int sn = nk % kStages;
      load_A(kc0 + nk, sn);
      if (!kNorm)
        load_B16(kc0 + nk, sn);
      else
        store_B(kc0 + nk, sn);
    }
    cp_async_commit();
  }
  cp_async_wait<0>();

  // ---- epilogue ----------------------------------------------------------------------------
  // acc[i][j]: m-tile wm + i, n-tile wn + j; c0/c1 -> weight row +lane/4, packed rows
  // 2(lane%4) + {0,1}; c2/c3 -> weight row +lane/4 + 8.
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const int mt = mt0 + wm + i;
    if (mt >= n_mt) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {      // packed row 2(lane%4) + h
        const int rr = (wn + j) * 8 + 2 * (lane & 3) + h;
        const int r = s_row[rr];
        if (r < 0) continue;
        const float v_lo = acc[i][j][h], v_hi = acc[i][j][2 + h];   // weight rows +lane/4, +lane/4 + 8
        const int o = mt * 16 + (lane >> 2);
        if (EPI == EPI_QKV) {
          a.out[(size_t)r * a.ld + o] = v_lo;
          a.out[(size_t)r * a.ld + o + 8] = v_hi;
        } else if (EPI == EPI_RESID) {   // k-slices of several CTAs add into the residual
          float* xr = a.out + (size_t)r * a.ld;
          atomicAdd(xr + o, v_lo);
          atomicAdd(xr + o + 8, v_hi);
        } else if (EPI == EPI_SWIGLU) {
          const int jj = mt * 8 + (lane >> 2);       // gate row (tile row lane/4), up row (+8)
          const float gt = v_lo;
          a.act[(size_t)r * a.ld + jj] = f32_to_bf16(gt / (1.0f + __expf(-gt)) * v_hi);
        } else {
          const int jd = s_j[rr];
          float* lg = a.logits + ((size_t)r * kRecSlots + jd) * a.V;
          float b0 = 0.f, b1 = 0.f;
          if (jd >= 1) {
            const float* bias = a.head_bias + ((size_t)(P - 1) * a.K + (jd - 1)) * a.V;
            b0 = __ldg(bias + o);
            b1 = __ldg(bias + o + 8);
          }
          lg[o] = v_lo + b0;
          lg[o + 8] = v_hi + b1;
        }
      }
    }
  }
}

// LM heads.  The (row, j) pairs of the call are grouped by head (head_list); group P starts at
// operand row qoff(P) = the sum of the earlier groups rounded up to 16 rows, and its columns
// are split into n_t = ceil(rows / kHeadTileMax) tiles of equal width (a multiple of 16), so
// every tile of the product belongs to one head and is no wider than the group needs.
constexpr int kHeadTileMax = 176;      // three 60 KB ring stages with the hi + lo operand
__device__ __forceinline__ int tc_head_qoff(const BatchInfo* info, int P) {
  int o = 0;
  for (int i = 1; i < P; ++i) o += (info->head_rows[i] + 15) / 16 * 16;
  return o;
}
__host__ __device__ __forceinline__ int tc_head_tiles(int rows) { return (rows + kHeadTileMax - 1) / kHeadTileMax; }
__host__ __device__ __forceinline__ int tc_head_width(int rows) {
  const int nt = tc_head_tiles(rows);
  return nt ? ((rows + nt - 1) / nt + 15) / 16 * 16 : 0;
}
// Grid bound over the tiles of every group: at most (K + 1) pairs per packed row.
inline int tc_head_grid_x(int R, int K, int n_pos) { return (R * (K + 1) + kHeadTileMax - 1) / kHeadTileMax + n_pos; }

// The pairs' normalised rows (final RMSNorm, hi + lo) as SW128 tiles of Qcap rows.
__global__ void __launch_bounds__(256) tc_heads_operand_kernel(const float* __restrict__ X, const float* __restrict__ gain,
                                                               const float* __restrict__ ss, int H, float eps,
                                                               const BatchInfo* info, const int* __restrict__ head_list,
                                                               int n_pos, int Qcap, uint8_t* hi, uint8_t* lo) {
  __shared__ int s_off[16], s_rows[16], s_q[16];
  if (threadIdx.x < 16) {
    const int P = threadIdx.x;
    s_off[P] = info->head_off[P];
    s_rows[P] = P >= 1 && P <= n_pos ? info->head_rows[P] : 0;
    s_q[P] = P >= 1 && P <= n_pos ? tc_head_qoff(info, P) : 0;
  }
  __syncthreads();
  const int T = info->n_pairs, cpr = H / 8;
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < T * cpr; i += gridDim.x * blockDim.x) {
    const int gi = i / cpr, ch = i - gi * cpr, k = ch * 8;
    int P = 1;
    while (P < n_pos && !(gi >= s_off[P] && gi < s_off[P] + s_rows[P])) ++P;
    const int q = s_q[P] + (gi - s_off[P]);
    const int r = head_list[gi] >> 3;
    const float s = rsqrtf(ss[r] / (float)H + eps);
    const float4 x0 = __ldcg(reinterpret_cast<const float4*>(X + (size_t)r * H + k));
    const float4 x1 = __ldcg(reinterpret_cast<const float4*>(X + (size_t)r * H + k + 4));
    const float4 g0 = __ldg(reinterpret_cast<const float4*>(gain + k));
    const float4 g1 = __ldg(reinterpret_cast<const float4*>(gain + k + 4));
    const float v[8] = {x0.x * g0.x * s, x0.y * g0.y * s, x0.z * g0.z * s, x0.w * g0.w * s,
                        x1.x * g1.x * s, x1.y * g1.y * s, x1.z * g1.z * s, x1.w * g1.w * s};
    uint32_t h[4], l[4];
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      h[t] = pack_bf16x2(v[2 * t], v[2 * t + 1]);
      l[t] = pack_bf16x2(v[2 * t] - bf16_lo_f32(h[t]), v[2 * t + 1] - bf16_hi_f32(h[t]));
    }
    const size_t off = tc::sw128_offset(Qcap, q, ch >> 3, ch & 7);
    *reinterpret_cast<uint4*>(hi + off) = make_uint4(h[0], h[1], h[2], h[3]);
    *reinterpret_cast<uint4*>(lo + off) = make_uint4(l[0], l[1], l[2], l[3]);
  }
}

// Logits of every pair: tile blockIdx.x (counted over the groups in head order) of head P's
// group times head P's weights (m-tile blockIdx.y), plus the draft-offset bias for j >= 1.
constexpr int kHeadsThreads = 256;     // eight warps: two per TMEM lane quarter in the epilogue
__global__ void __launch_bounds__(kHeadsThreads, 1) tc_heads_kernel(const tc::GemmArgs g, const uint8_t* w_heads,
                                                                    size_t head_bytes, float* logits,
                                                                    const float* head_bias, const BatchInfo* info,
                                                                    const int* head_list, int n_pos, int K, int V) {
  int P = 0, qoff = 0, c0 = 0, nw = 0, rows = 0;
  for (int i = 1, o = 0, t = blockIdx.x; i <= n_pos; ++i) {
    const int r = info->head_rows[i], nt = tc_head_tiles(r);
    if (P == 0 && t < nt) {
      const int w = tc_head_width(r);
      P = i;
      qoff = o;
      rows = r;
      c0 = t * w;
      nw = min(w, (r + 15) / 16 * 16 - c0);
    }
    t -= nt;
    o += (r + 15) / 16 * 16;
  }
  if (P == 0) return;                                   // past the last tile (uniform per CTA)
  const int off = info->head_off[P];
  // the tile's (row, j) entries in shared memory and this thread's bias of every offset j
  // (the epilogue's output row m is fixed per thread), loaded while the products run
  __shared__ int s_entry[kHeadTileMax];
  for (int i = threadIdx.x; i < nw; i += blockDim.x) s_entry[i] = c0 + i < rows ? head_list[off + c0 + i] : -1;
  const int m_t = blockIdx.y * tc::kBM + ((threadIdx.x >> 5) & 3) * 32 + (threadIdx.x & 31);
  float bias_j[kMaxDraft];
#pragma unroll
  for (int q = 0; q < kMaxDraft; ++q)
    bias_j[q] = q < K ? __ldg(head_bias + ((size_t)(P - 1) * K + q) * V + m_t) : 0.f;
  tc::GemmArgs ga = g;
  ga.a = w_heads + (size_t)(P - 1) * head_bytes;
  ga.n_active = nullptr;
  const int q0 = qoff + c0;
  tc::gemm_tile<kHeadTileMax, false, true>(
      ga,
      [&](int m, int n, float v, float) {
        const int e = s_entry[n - q0];
        if (e >= 0) {
          const int r = e >> 3, j = e & 7;
          float bias = 0.f;
#pragma unroll
          for (int q = 1; q <= kMaxDraft; ++q)
            if (j == q) bias = bias_j[q - 1];
          logits[((size_t)r * kRecSlots + j) * V + m] = v + bias;
        }
      },
      q0, nw);
}

// Per-row sums of squares of the residual stream after a residual GEMM (one warp per row):
// the next RMSNorm's 1/rms, applied while the next GEMM stages its operand.
__global__ void __launch_bounds__(256) batch_rowss_kernel(const float* X, int H, float* ss, const BatchInfo* info) {
  const int r = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (r >= info->M) return;
  const float4* x = reinterpret_cast<const float4*>(X + (size_t)r * H);
  float s = 0.f;
  for (int i = lane; i < (H >> 2); i += 32) {
    const float4 v = __ldcg(x + i);
    s += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
  if (lane == 0) ss[r] = s;
}

// ------------------------------------------------------------------------------------
// attention: one CTA per (stream, KV head).  At most 32 registers per thread, so that seven
// CTAs share an SM and the 1024 CTAs of 128 streams run as one wave.
// ------------------------------------------------------------------------------------
// Attention of the call's rows of stream s = blockIdx.x for KV head g = blockIdx.y and its
// `group` query heads (QK-norm, RoPE, causal softmax over the stream's cached positions and
// its new rows); outputs to the Wo product's operand.  Phases, with block barriers between
// them: (A) every input (the nr x group query vectors, cached and new K / V rows, RoPE rows
// of the new positions, QK-norm gains) copied into shared memory as 16-byte cp.async chunks,
// all in flight; (B) one warp per new q / k vector applies QK-norm and RoPE in registers and
// stores the new rows' K / V to the cache; (C) one warp per query vector: lanes 2j, 2j + 1
// score key j over interleaved chunks, softmax across the warp, then four output dims per
// lane summed over the keys.  Row and head of a query vector come from a table, not a
// division.
__global__ void __launch_bounds__(256, 7) batch_attn_kernel(FrameParams p, BatchBufs b, int layer) {
  const int s = blockIdx.x, g = blockIdx.y;
  if (s >= b.frame->S) return;
  const int base = b.sbase[s];
  if (base < 0) return;
  const DevState* st = p.st + s;
  const int nr = st->n_rows, pos0 = st->pos0;
  const int D = p.D, half = D >> 1, group = p.NH / p.NKV, nq = nr * group;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int lg4 = D == 128 ? 5 : 4, D4 = 1 << lg4;                // 16-byte chunks per row
  __shared__ __align__(16) float qs[kBatchQVec][132];
  __shared__ __align__(16) float ks[kBatchKeys][132];
  __shared__ __align__(16) float vs[kBatchKeys][128];
  __shared__ __align__(16) float2 cs[kMaxRows][64];               // RoPE (cos, sin) of the new rows
  __shared__ __align__(16) float gq[128], gk[128];
  __shared__ int q_row[kBatchQVec], q_head[kBatchQVec];
  const size_t cache_off = (size_t)s * p.kv_stride + ((size_t)layer * p.NKV + g) * p.kv_slots * D;
  const int nk = pos0 + nr;
  if (tid < nq) {
    q_row[tid] = tid / group;
    q_head[tid] = g * group + tid % group;
  }
  __syncthreads();
  // ---- (A) loads ----------------------------------------------------------------------
  {
    const int e_q = nq << lg4, e_k = e_q + (nk << lg4), e_v = e_k + (nk << lg4);
    const int e_cs = e_v + (nr << lg4), e_g = e_cs + (p.qk_norm ? 2 << lg4 : 0);
    for (int i = tid; i < e_g; i += 256) {
      const int ch = i & (D4 - 1);
      const float* src;
      float* dst;
      if (i < e_q) {
        const int qi = i >> lg4;
        src = b.qkv + (size_t)(base + q_row[qi]) * p.qkv_dim + q_head[qi] * D;
        dst = qs[qi];
      } else if (i < e_v) {
        const bool isv = i >= e_k;
        const int j = (i - (isv ? e_k : e_q)) >> lg4;
        if (j < pos0)
          src = (isv ? p.vcache : p.kcache) + cache_off + (size_t)j * D;
        else
          src = b.qkv + (size_t)(base + j - pos0) * p.qkv_dim + p.NH * D + (isv ? p.NKV * D : 0) + g * D;
        dst = isv ? vs[j] : ks[j];
      } else if (i < e_cs) {
        const int n = (i - e_v) >> lg4;
        src = reinterpret_cast<const float*>(p.rope + (size_t)(pos0 + n) * half);
        dst = reinterpret_cast<float*>(cs[n]);
      } else {
        const int w = (i - e_cs) >> lg4;
        src = (w == 0 ? p.q_norm : p.k_norm) + (size_t)layer * D;
        dst = w == 0 ? gq : gk;
      }
      cpa16(dst + 4 * ch, src + 4 * ch);
    }
    cpa_wait_all();
  }
  __syncthreads();
  // ---- (B) QK-norm + RoPE of the queries and the new keys; new K / V cached --------------
  const int nd = D >> 5;
  for (int vi = warp; vi < nq + nr; vi += 8) {
    const bool isq = vi < nq;
    const int n = isq ? q_row[vi] : vi - nq;
    float* row = isq ? qs[vi] : ks[pos0 + n];
    float x[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) x[i] = i < nd ? row[lane + 32 * i] : 0.f;
    if (p.qk_norm) {
      float ss = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) ss += x[i] * x[i];
#pragma unroll
      for (int off = 16; off; off >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, off);
      const float scl = rsqrtf(ss / (float)D + p.eps);
      const float* gg = isq ? gq : gk;
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (i < nd) x[i] = x[i] * scl * gg[lane + 32 * i];
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      if (i < nd / 2) {
        const float2 r = cs[n][lane + 32 * i];
        const float a0 = x[i], b0 = x[i + nd / 2];
        x[i] = a0 * r.x - b0 * r.y;
        x[i + nd / 2] = b0 * r.x + a0 * r.y;
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (i < nd) row[lane + 32 * i] = x[i];
    if (!isq) {
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (i < nd) {
          p.kcache[cache_off + (size_t)(pos0 + n) * D + lane + 32 * i] = x[i];
          p.vcache[cache_off + (size_t)(pos0 + n) * D + lane + 32 * i] = vs[pos0 + n][lane + 32 * i];
        }
    }
  }
  __syncthreads();
  // ---- (C) one warp per query vector: scores (lanes 2j, 2j+1), softmax, P.V ---------------
  const float scale = rsqrtf((float)D);
  for (int qi = warp; qi < nq; qi += 8) {
    const int n = q_row[qi], h = q_head[qi], npos = pos0 + n + 1;
    const int j = lane >> 1, hf = lane & 1;
    const bool live = j < npos;                      // causal: keys 0..pos0+n
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
    if (live) {
      const float4* q4 = reinterpret_cast<const float4*>(qs[qi]) + hf;
      const float4* k4 = reinterpret_cast<const float4*>(ks[j]) + hf;
#pragma unroll 4
      for (int c2 = 0; c2 < (D4 >> 1); ++c2) {
        const float4 q = q4[2 * c2], k = k4[2 * c2];
        a0 += q.x * k.x;
        a1 += q.y * k.y;
        a2 += q.z * k.z;
        a3 += q.w * k.w;
      }
    }
    float sc = (a0 + a1) + (a2 + a3);
    sc += __shfl_xor_sync(0xFFFFFFFFu, sc, 1);
    sc = live ? sc * scale : -INFINITY;
    float mx = sc;
#pragma unroll
    for (int off = 16; off > 1; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xFFFFFFFFu, mx, off));
    const float e = live ? __expf(sc - mx) : 0.f;
    float sum = e;                                   // lanes of one parity hold every key once
#pragma unroll
    for (int off = 16; off > 1; off >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, off);
    const float pj = e / sum;
    const int d0 = 4 * lane;                         // four dims per lane
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int jj = 0; jj < npos; ++jj) {
      const float w = __shfl_sync(0xFFFFFFFFu, pj, 2 * jj);
      if (d0 < D) {
        const float4 v = *reinterpret_cast<const float4*>(&vs[jj][d0]);
        acc.x += w * v.x;
        acc.y += w * v.y;
        acc.z += w * v.z;
        acc.w += w * v.w;
      }
    }
    if (d0 < D) {
      const int f = h * D + d0;
      const uint2 packed = make_uint2(pack_bf16x2(acc.x, acc.y), pack_bf16x2(acc.z, acc.w));
      if (b.att_t)        // the Wo product's operand, SW128 tiles (tensor-core path)
        *reinterpret_cast<uint2*>(b.att_t + tc::sw128_offset(b.Rtc, base + n, f >> 6, (f & 63) >> 3) + (f & 7) * 2) =
            packed;
      else
        *reinterpret_cast<uint2*>(b.att + (size_t)(base + n) * p.NH * D + f) = packed;
    }
  }
}

// ------------------------------------------------------------------------------------
// top-k of every (row, j) distribution of the call; then the acceptance per stream
// ------------------------------------------------------------------------------------
__global__ void __launch_bounds__(kConsumerThreads) batch_topk_kernel(FrameParams p, BatchBufs b, int call) {
  __shared__ __align__(16) uint8_t smem_raw[sizeof(TopkScratch)];
  TopkScratch& ts = *reinterpret_cast<TopkScratch*>(smem_raw);
  if ((int)blockIdx.x >= b.info->n_pairs) return;
  const int e = b.pairs[blockIdx.x], r = e >> 3, j = e & 7;
  const int greedy = (j > 0 && p.draft_mode == MCD_DRAFT_GREEDY) ? 1 : 0;
  TopkRec* recs = b.recs + (size_t)(call & 1) * b.R * kRecSlots;
  block_topk(b.logits + ((size_t)r * kRecSlots + j) * p.V, p.V, p.top_k, p.T, greedy, ts,
             recs + (size_t)r * kRecSlots + j);
}

__global__ void __launch_bounds__(kConsumerThreads) batch_accept_kernel(FrameParams p, BatchBufs b, int call) {
  const int s = blockIdx.x;
  const BatchFrame* fa = b.frame;
  if (s >= fa->S) return;
  const int base = b.sbase[s];
  if (base < 0) return;
  DevState* st = p.st + s;
  __shared__ AcceptResult s_res;
  __shared__ int s_next[kMaxDraft], s_old[kMaxDraft + 1];
  const int a = st->a, n_d = st->n_d, pos0 = st->pos0, n_rows = st->n_rows, qrow = st->q_row;
  const int fr = st->first_head_row;
  if (threadIdx.x <= kMaxDraft) s_old[threadIdx.x] = (int)threadIdx.x < n_d ? st->drafts[threadIdx.x] : -1;
  __syncthreads();
  const unsigned sid = fa->stream_ids[s], fid = fa->frame_ids[s];
  const TopkRec* cur = b.recs + (size_t)(call & 1) * b.R * kRecSlots;
  const TopkRec* prev = b.recs + (size_t)((call + 1) & 1) * b.R * kRecSlots;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // every record the acceptance reads, staged in shared memory first: p of positions
  // a+1 .. (the bonus row only when its position exists), then q of the drafts
  __shared__ __align__(16) TopkRec srec[2 * kMaxDraft + 1];
  const int n_p = a + 1 + n_d <= p.P ? n_d + 1 : n_d;
  stage_records(srec, n_p + n_d, p.top_k, [&](int r) {
    return r < n_p ? cur + (size_t)(base + a + 1 + r - pos0) * kRecSlots : prev + (size_t)qrow * kRecSlots + 1 + (r - n_p);
  });
  __syncthreads();
  // every draft's accept test and the residual draw it would take as the first rejection in
  // parallel (warp i for draft i), warp n_d the bonus draw; then the chain is read off in
  // order, taking the same decisions as testing the drafts one after another
  __shared__ int s_ok[kMaxDraft + 1], s_alt[kMaxDraft + 1];
  if (warp <= n_d) {
    const int i = warp, pos = a + 1 + i;
    if (i < n_d) {
      const TopkRec* pr = srec + i;
      const TopkRec* qr = srec + n_p + i;
      const int d = s_old[i];
      const unsigned long long wp = warp_weight(pr, d), wq = warp_weight(qr, d);
      const unsigned long long U = uniform_U(p.seed, sid, fid, call, pos, PURPOSE_ACCEPT);
      const bool ok = lt128(mul128x64(mul64(U, wq), pr->S), shl53(wp * qr->S));
      const int alt = ok ? -1 : warp_residual(pr, qr, uniform_U(p.seed, sid, fid, call, pos, PURPOSE_TARGET));
      if (lane == 0) {
        s_ok[i] = ok ? 1 : 0;
        s_alt[i] = alt;
      }
    } else if (pos <= p.P) {
      const int bonus = warp_draw(srec + n_d, uniform_U(p.seed, sid, fid, call, pos, PURPOSE_TARGET));
      if (lane == 0) s_alt[i] = bonus;
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    AcceptResult r;
    r.n_acc = 0;
    r.n_emit = 0;
    bool rejected = false;
    for (int i = 0; i < n_d && !rejected; ++i) {
      if (s_ok[i]) {
        r.emitted[r.n_emit++] = s_old[i];
        ++r.n_acc;
      } else {
        r.emitted[r.n_emit++] = s_alt[i];
        rejected = true;
      }
    }
    if (!rejected && a + 1 + n_d <= p.P) r.emitted[r.n_emit++] = s_alt[n_d];
    s_res = r;
  }
  __syncthreads();
  const int n_emit = s_res.n_emit, n_acc = s_res.n_acc;
  const int a_new = a + n_emit, m = a_new - pos0, n_next = min(p.K, p.P - a_new);
  // next drafts from the draft distributions of row m, whose head emitted the last code
  stage_records(srec, n_next, p.top_k, [&](int r) { return cur + (size_t)(base + m) * kRecSlots + 1 + r; });
  __syncthreads();
  for (int j = 1 + warp; j <= n_next; j += kConsumerWarps) {
    const unsigned long long U = uniform_U(p.seed, sid, fid, call, a_new + j, PURPOSE_DRAFT);
    const int d = warp_draw(srec + (j - 1), U);
    if (lane == 0) s_next[j - 1] = d;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int* codes_out = fa->codes_out ? fa->codes_out + (size_t)s * p.P : nullptr;
    for (int t = 0; t < n_emit; ++t) {
      st->codes[a + 1 + t] = s_res.emitted[t];
      if (codes_out) codes_out[a + t] = s_res.emitted[t];
    }
    for (int j = 0; j < n_next; ++j) st->drafts[j] = s_next[j];
    for (int t = 0; t < n_emit; ++t) st->emitted_last[t] = s_res.emitted[t];
    const int p_lo = a + 1, p_hi = min(p.P, pos0 + n_rows - 1 + p.K);
    const int calls = st->calls + 1, heads = st->heads_read + p_hi - p_lo + 1;
    const int kvr = st->kv_rows + pos0 + n_rows, rf = st->rows_fed + n_rows;
    const int drafted = st->drafted + n_d, accepted = st->accepted + n_acc;
    st->n_emit_last = n_emit;
    st->n_acc_last = n_acc;
    st->a = a_new;
    st->n_d = n_next;
    st->pos0 = a_new + 1;
    st->n_rows = min(n_next + 1, p.P - a_new);
    st->top_pos = st->pos0 + st->n_rows - 1;
    st->round = call + 1;
    st->first_head_row = 0;
    st->calls = calls;
    st->heads_read = heads;
    st->kv_rows = kvr;
    st->rows_fed = rf;
    st->drafted = drafted;
    st->accepted = accepted;
    st->call = call + 1;
    st->done = a_new >= p.P ? 1 : 0;
    st->q_row = base + m;     // the next call's q: this call's records of packed row base + m
    if (a_new >= p.P && fa->stats) {
      mcd_frame_stats* fs = fa->stats + s;
      fs->calls = calls;
      fs->codes = a_new;
      fs->drafted = drafted;
      fs->accepted = accepted;
      fs->status = *(volatile int*)p.err;
      fs->heads_read = heads;
      fs->kv_rows = kvr;
      fs->rows_fed = rf;
    }
  }
  // optional trace, in the frame kernel's layout
  if (fa->trace && call < kMaxCalls) {
    uint8_t* tb = fa->trace + (size_t)s * p.trace_stride;
    mcd_call_trace* tr = reinterpret_cast<mcd_call_trace*>(tb) + call;
    if (threadIdx.x == 0) {
      tr->a = a;
      tr->n_rows = n_rows;
      tr->pos0 = pos0;
      tr->n_drafts = n_d;
      for (int n = 0; n < kMaxRows; ++n) tr->input_ids[n] = n < n_rows ? b.rows[base + n].id : -1;
      for (int i = 0; i < kMaxRows; ++i) tr->drafts[i] = i < n_d ? s_old[i] : -1;
      tr->n_acc = n_acc;
      tr->n_emit = n_emit;
      for (int t = 0; t < kMaxRows; ++t) tr->emitted[t] = t < n_emit ? s_res.emitted[t] : -1;
      tr->n_next = n_next;
      for (int j = 0; j < kMaxRows; ++j) tr->next_drafts[j] = j < n_next ? s_next[j] : -1;
      tr->draft_row = m;
    }
    float* vlog = reinterpret_cast<float*>(tb + sizeof(mcd_call_trace) * kMaxCalls);
    float* dlog = vlog + (size_t)kMaxCalls * kMaxRows * p.V;
    for (int idx = threadIdx.x; idx < kMaxRows * p.V; idx += blockDim.x) {
      const int n = idx / p.V, v = idx - n * p.V;
      if (n >= fr && n < n_rows)
        vlog[((size_t)call * kMaxRows + n) * p.V + v] = __ldcg(b.logits + ((size_t)(base + n) * kRecSlots) * p.V + v);
      if (n < n_next)
        dlog[((size_t)call * kMaxRows + n) * p.V + v] =
            __ldcg(b.logits + ((size_t)(base + m) * kRecSlots + n + 1) * p.V + v);
    }
  }
}

__global__ void batch_begin_kernel(FrameParams p, BatchBufs b) {
  const BatchFrame* fa = b.frame;
  for (int s = threadIdx.x; s < fa->S; s += blockDim.x) init_stream_state(p.st + s, p.C0V > 0 ? fa->c0[s] : -1);
}

}  // namespace mcd

// ------------------------------------------------------------------------------------
// Host side: buffers, the per-context graph, one launch per frame
// ------------------------------------------------------------------------------------
namespace mcd {

struct BatchState {
  BatchBufs b;
  BatchFrame host_frame;
  int max_streams = 0;
  bool use_tc = false;        // QKV, Wo, gate/up and down on the tcgen05 GEMM
  TcWeights tw;
  cudaGraph_t graph = nullptr;
  cudaGraphExec_t exec = nullptr;
  cudaStream_t cap = nullptr;
  std::vector<void*> allocs;
};

template <class T>
static cudaError_t batch_alloc(BatchState* bs, T** p, size_t bytes) {
  void* q = nullptr;
  cudaError_t e = cudaMalloc(&q, bytes < 256 ? 256 : bytes);
  if (e != cudaSuccess) return e;
  bs->allocs.push_back(q);
  *p = static_cast<T*>(q);
  return cudaSuccess;
}

void batch_destroy(BatchState* bs) {
  if (!bs) return;
  if (bs->exec) cudaGraphExecDestroy(bs->exec);
  if (bs->graph) cudaGraphDestroy(bs->graph);
  if (bs->cap) cudaStreamDestroy(bs->cap);
  for (void* q : bs->allocs) cudaFree(q);
  delete bs;
}

int batch_rows(const FrameParams& p, int max_streams) { return max_streams * std::max(p.K + 1, 2); }

// From 5 streams on, a launch the persistent frame kernel could take runs faster on the
// tensor-core batched path (measured on GB300: +10 % at 5 streams, +17 % at 8) when the
// shapes allow the tcgen05 GEMMs and one attention CTA holds a stream's query vectors.
bool batch_prefers(const FrameParams& p, int n_streams) {
  return n_streams >= kBatchMinStreams && tc_block_supported(p) &&
         std::max(p.K + 1, 2) * (p.NH / p.NKV) <= kBatchQVec && p.draft_mode != MCD_DRAFT_NOISY_TARGET &&
         p.draft_mode != MCD_DRAFT_TREE;
}

mcd_status batch_create(const FrameParams& p, int max_streams, BatchState** out) {
  *out = nullptr;
  BatchState* bs = new BatchState();
  bs->max_streams = max_streams;
  auto fail = [&](mcd_status s) {
    batch_destroy(bs);
    return s;
  };
  BatchBufs& b = bs->b;
  const int R = (batch_rows(p, max_streams) + kGN - 1) / kGN * kGN;
  b.R = R;
  cudaError_t e;
#define BATCH_ALLOC(ptr, bytes)                                                        \
  do {                                                                                 \
    if ((e = batch_alloc(bs, &(ptr), (bytes))) != cudaSuccess) return fail(cuda_status(e)); \
  } while (0)
  BATCH_ALLOC(b.info, sizeof(BatchInfo));
  BATCH_ALLOC(b.frame, sizeof(BatchFrame));
  BATCH_ALLOC(b.rows, sizeof(BatchRow) * R);
  BATCH_ALLOC(b.sbase, sizeof(int) * kMaxBatchStreams);
  BATCH_ALLOC(b.pairs, sizeof(int) * R * kRecSlots);
  BATCH_ALLOC(b.head_list, sizeof(int) * R * kRecSlots);
  BATCH_ALLOC(b.X, sizeof(float) * R * p.H);
  BATCH_ALLOC(b.ss, sizeof(float) * (2 * p.L + 1) * R);
  BATCH_ALLOC(b.qkv, sizeof(float) * R * p.qkv_dim);
  BATCH_ALLOC(b.att, sizeof(uint16_t) * R * p.NH * p.D);
  BATCH_ALLOC(b.act, sizeof(uint16_t) * R * p.F);
  BATCH_ALLOC(b.logits, sizeof(float) * R * kRecSlots * p.V);
  BATCH_ALLOC(b.recs, sizeof(TopkRec) * 2 * R * kRecSlots);
  bs->use_tc = tc_block_supported(p);
  if (bs->use_tc) {
    const int Rtc = (R + 127) / 128 * 128;
    b.Rtc = Rtc;
    BATCH_ALLOC(b.xn_hi, (size_t)Rtc * p.H * 2);
    BATCH_ALLOC(b.xn_lo, (size_t)Rtc * p.H * 2);
    BATCH_ALLOC(b.att_t, (size_t)Rtc * p.NH * p.D * 2);
    BATCH_ALLOC(b.act_t, (size_t)Rtc * p.F * 2);
    BATCH_ALLOC(b.part, (size_t)kTcSplit * Rtc * p.H * 4);
    if (p.V % tc::kBM == 0) {
      b.Qcap = (R * kRecSlots + p.P * (kTcBN - 1) + kTcBN - 1) / kTcBN * kTcBN;
      BATCH_ALLOC(b.hq_hi, (size_t)b.Qcap * p.H * 2);
      BATCH_ALLOC(b.hq_lo, (size_t)b.Qcap * p.H * 2);
      BATCH_ALLOC(bs->tw.heads, (size_t)p.P * p.V * p.H * 2);
    }
    TcWeights& tw = bs->tw;
    tw.off = tc_layer_offsets(p);
    BATCH_ALLOC(tw.arena, tw.off.layer * p.L);
  }
#undef BATCH_ALLOC
  if (cudaMemset(b.info, 0, sizeof(BatchInfo)) != cudaSuccess) return fail(MCD_ERR_CUDA);
  if (cudaStreamCreateWithFlags(&bs->cap, cudaStreamNonBlocking) != cudaSuccess) return fail(MCD_ERR_CUDA);
  void* gemms[] = {(void*)batch_gemm_kernel<BSRC_NORM_HILO, EPI_QKV>, (void*)batch_gemm_kernel<BSRC_BF16, EPI_RESID>,
                   (void*)batch_gemm_kernel<BSRC_NORM, EPI_SWIGLU>, (void*)batch_gemm_kernel<BSRC_NORM_HILO, EPI_HEADS>};
  for (void* fn : gemms)
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kGemmSmemHilo) != cudaSuccess)
      return fail(MCD_ERR_CUDA);
  if (bs->use_tc &&
      (tc_block_set_smem() != cudaSuccess ||
       cudaFuncSetAttribute(tc_heads_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                            tc::Layout<kHeadTileMax, false, true>::kSmemBytes) != cudaSuccess))
    return fail(MCD_ERR_CUDA);
  *out = bs;
  return MCD_OK;
}

// The tcgen05 GEMMs' copies of layer l's matrices (row-major bf16 sources, device).
mcd_status batch_load_layer(BatchState* bs, const FrameParams& p, cudaStream_t st, const LayerSrc& src, int l) {
  if (!bs || !bs->use_tc) return MCD_OK;
  tc_tile_layer(p, st, src.wq, src.wk, src.wv, src.wo, src.wg, src.wu, src.wd, bs->tw.arena + (size_t)l * bs->tw.off.layer);
  return cudaGetLastError() == cudaSuccess ? MCD_OK : MCD_ERR_CUDA;
}

// The tcgen05 GEMM's copy of LM head P (row-major bf16 [V][H] source, device).
mcd_status batch_load_head(BatchState* bs, const FrameParams& p, cudaStream_t st, const uint8_t* src, int P) {
  if (!bs || !bs->tw.heads) return MCD_OK;
  tc_weight_tile_kernel<<<512, 256, 0, st>>>(reinterpret_cast<const uint16_t*>(src), p.V, p.H, p.V, 0, p.V, 0,
                                             bs->tw.heads + (size_t)(P - 1) * p.V * p.H * 2);
  return cudaGetLastError() == cudaSuccess ? MCD_OK : MCD_ERR_CUDA;
}

static GemmArgs gemm_args(const FrameParams& p, const BatchBufs& b) {
  GemmArgs a;
  memset(&a, 0, sizeof(a));
  a.info = b.info;
  a.head_list = b.head_list;
  a.eps = p.eps;
  a.K = p.K;
  a.V = p.V;
  return a;
}

// k-slices of a residual GEMM: enough CTAs for about two per SM, at least 4 k-chunks each.
static int split_k(dim3 grid, int K, int n_sm) {
  const int ctas = (int)(grid.x * grid.y), chunks = K / kGK;
  int z = 1;
  while (ctas * z < 2 * n_sm && chunks / (2 * z) >= 4) z *= 2;
  return z;
}

// Every kernel of one frame, in stream order on `s` (captured into the graph).
static cudaError_t enqueue_frame(const FrameParams& p, const BatchState* bs, cudaStream_t s) {
  const BatchBufs& b = bs->b;
  const int R = b.R, L = p.L, H = p.H;
  const dim3 blk(256);
  batch_begin_kernel<<<1, 256, 0, s>>>(p, b);
  for (int call = 0; call < p.P; ++call) {
    batch_pack_kernel<<<1, 256, 0, s>>>(p, b);
    batch_embed_kernel<<<R, 256, 0, s>>>(p, b);
    for (int l = 0; l < L && bs->use_tc; ++l) {
      const uint8_t* wl = bs->tw.arena + (size_t)l * bs->tw.off.layer;
      const int Rtc = b.Rtc, qd = p.NH * p.D;
      const dim3 pblk(tc::kPThreads);
      // RMSNorm -> QKV (hi + lo operand; after layer 0 written by the previous layer's last
      // residual pass)
      if (l == 0)
        tc_norm_operand_kernel<<<256, blk, 0, s>>>(b.X, p.attn_norm, b.ss, H, p.eps, &b.info->M, Rtc, b.xn_hi, b.xn_lo);
      {
        const tc::GemmArgs g{wl + bs->tw.off.qkv, nullptr, b.xn_hi, b.xn_lo, p.qkv_dim, Rtc, H, &b.info->M, p.err, p.wait_ns};
        tc_qkv_kernel<<<tc_grid(tc_tiles(Rtc, kTcBN, p.qkv_dim, 1), p.n_cta), pblk, tc::PLayout<kTcBN, false, true>::kSmemBytes, s>>>(
            g, b.qkv, p.qkv_dim, &b.info->M);
      }
      batch_attn_kernel<<<dim3(bs->max_streams, p.NKV), blk, 0, s>>>(p, b, l);      // -> att_t
      // Wo (k-split partials) -> residual, ss, the gate/up operand
      tc_launch_resid(wl + bs->tw.off.o, b.att_t, b.part, H, Rtc, qd, &b.info->M, p.err, p.wait_ns, p.n_cta, s);
      tc_resid_norm_kernel<<<R, 128, 0, s>>>(b.X, b.part, tc_splits(qd, tc_resid_split(Rtc)), Rtc, H, &b.info->M, b.ss + (size_t)(2 * l + 1) * R,
                                             p.ffn_norm + (size_t)l * H, p.eps, b.xn_hi, nullptr);
      // gate/up -> SwiGLU (into the down product's operand)
      tc_launch_gu(wl + bs->tw.off.gu, b.xn_hi, b.act_t, Rtc, &b.info->M, p.F, H, p.err, p.wait_ns, p.n_cta, s);
      // down (k-split partials) -> residual, ss, the next layer's QKV operand
      tc_launch_resid(wl + bs->tw.off.d, b.act_t, b.part, H, Rtc, p.F, &b.info->M, p.err, p.wait_ns, p.n_cta, s);
      const bool last = l + 1 == L;
      tc_resid_norm_kernel<<<R, 128, 0, s>>>(b.X, b.part, tc_splits(p.F, tc_resid_split(Rtc)), Rtc, H, &b.info->M, b.ss + (size_t)(2 * l + 2) * R,
                                             last ? nullptr : p.attn_norm + (size_t)(l + 1) * H, p.eps, b.xn_hi, b.xn_lo);
    }
    for (int l = 0; l < L && !bs->use_tc; ++l) {
      {   // RMSNorm -> QKV
        GemmArgs a = gemm_args(p, b);
        a.W = p.w_qkv + (size_t)l * p.g[MAT_QKV].stride;
        a.g = p.g[MAT_QKV];
        a.X = b.X;
        a.ldx = H;
        a.gain = p.attn_norm + (size_t)l * H;
        a.ss = b.ss + (size_t)(2 * l) * R;
        a.out = b.qkv;
        a.ld = p.qkv_dim;
        batch_gemm_kernel<BSRC_NORM_HILO, EPI_QKV>
            <<<dim3(a.g.M / kGM + (a.g.M % kGM != 0), R / kGN), blk, kGemmSmemHilo, s>>>(a);
      }
      batch_attn_kernel<<<dim3(bs->max_streams, p.NKV), blk, 0, s>>>(p, b, l);
      {   // Wo + residual
        GemmArgs a = gemm_args(p, b);
        a.W = p.w_wo + (size_t)l * p.g[MAT_WO].stride;
        a.g = p.g[MAT_WO];
        a.Xb = b.att;
        a.ldx = p.NH * p.D;
        a.out = b.X;
        a.ld = H;
        const dim3 grid(a.g.M / kGM + (a.g.M % kGM != 0), R / kGN);
        batch_gemm_kernel<BSRC_BF16, EPI_RESID><<<dim3(grid.x, grid.y, split_k(grid, a.g.K, p.n_cta)), blk, kGemmSmem, s>>>(a);
        batch_rowss_kernel<<<R / 8, blk, 0, s>>>(b.X, H, b.ss + (size_t)(2 * l + 1) * R, b.info);
      }
      {   // RMSNorm -> gate/up -> SwiGLU
        GemmArgs a = gemm_args(p, b);
        a.W = p.w_gu + (size_t)l * p.g[MAT_GU].stride;
        a.g = p.g[MAT_GU];
        a.X = b.X;
        a.ldx = H;
        a.gain = p.ffn_norm + (size_t)l * H;
        a.ss = b.ss + (size_t)(2 * l + 1) * R;
        a.act = b.act;
        a.ld = p.F;
        batch_gemm_kernel<BSRC_NORM, EPI_SWIGLU><<<dim3(a.g.M / kGM + (a.g.M % kGM != 0), R / kGN), blk, kGemmSmem, s>>>(a);
      }
      {   // down + residual
        GemmArgs a = gemm_args(p, b);
        a.W = p.w_wd + (size_t)l * p.g[MAT_WD].stride;
        a.g = p.g[MAT_WD];
        a.Xb = b.act;
        a.ldx = p.F;
        a.out = b.X;
        a.ld = H;
        const dim3 grid(a.g.M / kGM + (a.g.M % kGM != 0), R / kGN);
        batch_gemm_kernel<BSRC_BF16, EPI_RESID><<<dim3(grid.x, grid.y, split_k(grid, a.g.K, p.n_cta)), blk, kGemmSmem, s>>>(a);
        batch_rowss_kernel<<<R / 8, blk, 0, s>>>(b.X, H, b.ss + (size_t)(2 * l + 2) * R, b.info);
      }
    }
    if (bs->tw.heads) {   // final RMSNorm -> LM heads on the tensor cores, tiles grouped by head
      tc_heads_operand_kernel<<<512, blk, 0, s>>>(b.X, p.final_norm, b.ss + (size_t)(2 * L) * R, H, p.eps, b.info,
                                                 b.head_list, p.P, b.Qcap, b.hq_hi, b.hq_lo);
      const tc::GemmArgs g{nullptr, nullptr, b.hq_hi, b.hq_lo, p.V, b.Qcap, H, nullptr, p.err, p.wait_ns};
      tc_heads_kernel<<<dim3(tc_head_grid_x(R, p.K, p.P), p.V / tc::kBM, 1), dim3(kHeadsThreads),
                        tc::Layout<kHeadTileMax, false, true>::kSmemBytes, s>>>(g, bs->tw.heads, (size_t)p.V * H * 2, b.logits,
                                                                        p.head_bias, b.info, b.head_list, p.P, p.K, p.V);
    } else {   // final RMSNorm -> LM heads, one grid slice per head
      GemmArgs a = gemm_args(p, b);
      a.W = p.w_head;
      a.g = p.g[MAT_HEAD];
      a.X = b.X;
      a.ldx = H;
      a.gain = p.final_norm;
      a.ss = b.ss + (size_t)(2 * L) * R;
      a.logits = b.logits;
      a.head_bias = p.head_bias;
      batch_gemm_kernel<BSRC_NORM_HILO, EPI_HEADS>
          <<<dim3(a.g.M / kGM + (a.g.M % kGM != 0), R / kGN, p.P), blk, kGemmSmemHilo, s>>>(a);
    }
    batch_topk_kernel<<<R * (p.K + 1), kConsumerThreads, 0, s>>>(p, b, call);
    batch_accept_kernel<<<bs->max_streams, kConsumerThreads, 0, s>>>(p, b, call);
  }
  return cudaGetLastError();
}

mcd_status batch_decode(BatchState* bs, const FrameParams& p, cudaStream_t stream, int n, const uint32_t* stream_ids,
                        const uint32_t* frame_ids, const float* cond, const int32_t* c0, const float* c0_emb,
                        int32_t* codes_out, mcd_frame_stats* stats, uint8_t* trace) {
  if (n < 1 || n > bs->max_streams) return MCD_ERR_INVALID_ARG;
  if (!bs->exec) {
    cudaStream_t s = bs->cap;
    MCD_CHECK(cudaStreamBeginCapture(s, cudaStreamCaptureModeThreadLocal));
    cudaError_t e = enqueue_frame(p, bs, s);
    cudaGraph_t g = nullptr;
    cudaError_t e2 = cudaStreamEndCapture(s, &g);
    if (e != cudaSuccess || e2 != cudaSuccess) {
      if (g) cudaGraphDestroy(g);
      return cuda_status(e != cudaSuccess ? e : e2);
    }
    bs->graph = g;
    MCD_CHECK(cudaGraphInstantiate(&bs->exec, g, 0));
  }
  BatchFrame& f = bs->host_frame;
  memset(&f, 0, sizeof(f));
  f.S = n;
  for (int i = 0; i < n; ++i) {
    f.stream_ids[i] = stream_ids[i];
    f.frame_ids[i] = frame_ids[i];
  }
  f.cond = cond;
  f.c0 = c0;
  f.c0emb = c0_emb;
  f.codes_out = codes_out;
  f.stats = stats;
  f.trace = trace;
  MCD_CHECK(cudaMemcpyAsync(bs->b.frame, &f, sizeof(f), cudaMemcpyHostToDevice, stream));
  MCD_CHECK(cudaGraphLaunch(bs->exec, stream));
  return MCD_OK;
}

}  // namespace mcd
