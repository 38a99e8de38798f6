// Internal definitions of libmcd: device-side structures, limits and PTX helpers.
//
// Data layout in HBM (one context = one stream's model + state):
//   * Weight matrices of the hot path are stored as "units": a unit is Mu x Ku tiles of
//     16 x 16 elements, contiguous, so one bulk copy moves one unit into a shared-memory
//     ring slot.  A bf16 tile is 512 B in the A-fragment order of mma.m16n8k16 (lane l
//     holds rows l/4 and l/4+8, columns 2(l%4)+{0,1} and +8), an fp32 tile is 1 KB with
//     lane l holding row l%16, columns 8*(l/16)..+7.  Units of a matrix are ordered
//     [k-chunk][m-block]; tiles inside a unit [m-tile][k-tile].
//   * Embedding tables stay row-major [vocab, hidden] in the weight dtype (row gather).
//   * Norm gains and offsets are fp32.  Activations, KV cache and logits are fp32.
//   * W8A16 (MCD_WEIGHT_INT8): the same tiles with one byte per element (256 B per tile, in
//     the bf16 tile's element order) and one fp32 scale per output row; the unit GEMMs widen
//     the bytes to bf16 in registers and the epilogues apply the row scale.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>
#include "../../include/mcd.h"

namespace mcd {

constexpr int kMaxRows = 8;          // rows of one stream in one call (K + 1 <= 8; first call uses 2)
constexpr int kMaxCols = 32;         // rows of one call over all streams (packed operand columns)
constexpr int kMaxStreams = 8;       // streams decoded together by one launch of the frame kernel
constexpr int kMaxBatchStreams = 128;  // streams of one batched decode (GEMM path)
constexpr int kMaxBatchRows = 512;     // packed rows of one batched call
constexpr int kMaxDraft = 7;         // K
constexpr int kMaxTopK = 128;
constexpr int kMaxPos = 32;          // KV positions kept per frame (cond, c0, c1..c14 used)
constexpr int kMaxTree = 64;         // tree nodes (a tree call feeds 1 + nodes rows)
constexpr int kMaxTreeRows = kMaxTree + 1;
constexpr int kTreeKeys = 48;        // keys of one tree attention task (prefix + visible rows)
constexpr int kMaxTreeRank = 8;      // candidates per drafted position
constexpr int kMaxCalls = 16;        // verify calls per frame (15 positions, first call emits 1)
constexpr int kMaxSlots = 128;       // passes per frame: verify calls + noisy-target drafting passes
constexpr int kMaxVocab = 4096;
constexpr int kConsumerWarps = 8;
constexpr int kConsumerThreads = kConsumerWarps * 32;
constexpr int kThreads = kConsumerThreads + 32;   // + one producer warp
constexpr int kSlotBytes = 32768;
constexpr int kNumSlots = 4;
constexpr int kChunk = 3;            // units of one stage multiplied before one epilogue pass (<= kNumSlots)
constexpr int kActBytes = 32768;     // fp32 activation rows / attention / top-k scratch
constexpr int kBfragBytes = 32768;   // B operand (activations) of the unit GEMMs
constexpr int kRedBytes = 16384;     // cross-warp partial tiles of a chunk of units

enum MatKind { MAT_QKV = 0, MAT_WO = 1, MAT_GU = 2, MAT_WD = 3, MAT_HEAD = 4, MAT_COUNT = 5 };

struct MatGeom {
  int M, K;            // logical rows / columns
  int Mu, Ku;          // m-tiles and k-tiles per unit
  int n_mb, n_kc;      // m-blocks, k-chunks
  int n_units;         // n_mb * n_kc
  int unit_bytes;
  long long stride;    // bytes between consecutive matrices of this kind (layer / head)
};

// Per-call state shared by all CTAs, rewritten by the CTA that runs the acceptance step.
struct DevState {
  int call;            // slot (counter set) of the next pass: every verify call and every
                       // noisy-target drafting pass takes one
  int a;               // codes emitted so far
  int done;
  int n_d;             // pending drafts (positions a+1..a+n_d)
  int pos0;            // sequence position of the next call's first row
  int n_rows;          // rows of the next call
  int first_head_row;  // first row that reads an LM head (1 in the first call)
  int n_acc_last;
  int q_row;           // row of the previous call whose draft records are pending
  int codes[kMaxPos];  // codes[0] = c0 id (or -1), codes[s] = c_s
  int drafts[kMaxDraft + 1];
  int emitted_last[kMaxRows];
  int n_emit_last;
  int calls, drafted, accepted;
  int heads_read;      // LM heads streamed, summed over the frame's calls
  int kv_rows;         // sum over calls of (pos0 + n_rows): KV positions read or written
  int rows_fed;        // sum over calls of n_rows
  int err;
  int round;           // verify round of the next pass (Philox round, trace index)
  int emu;             // 0: the next pass is a verify call; j >= 1: noisy-target pass j
  int tpass;           // TREE mode: pass of the next call (rows 32 t .. 32 t + 31 of the call)
  int emu_n;           // drafts the noisy-target passes make for the next verify call
  int emu_in;          // code fed to the next noisy-target pass
  int top_pos;         // largest row position of the next pass
};

// State of a stream at the start of a frame: the first call feeds [cond, c0] (positions 0, 1).
__device__ inline void init_stream_state(DevState* st, int c0) {
  st->call = 0;
  st->a = 0;
  st->done = 0;
  st->n_d = 0;
  st->pos0 = 0;
  st->n_rows = 2;
  st->first_head_row = 1;
  st->n_acc_last = 0;
  st->q_row = 0;
  st->round = 0;
  st->emu = 0;
  st->tpass = 0;
  st->emu_n = 0;
  st->emu_in = -1;
  st->top_pos = 1;
  for (int i = 0; i < kMaxPos; ++i) st->codes[i] = -1;
  st->codes[0] = c0;
  for (int i = 0; i <= kMaxDraft; ++i) st->drafts[i] = -1;
  st->n_emit_last = 0;
  st->calls = st->drafted = st->accepted = 0;
  st->heads_read = st->kv_rows = st->rows_fed = 0;
}

// One top-k / temperature distribution as integer weights: p(ids[i]) = W[i] / S.
struct TopkRec {
  int n;
  int pad;
  unsigned long long S;
  int ids[kMaxTopK];
  uint32_t W[kMaxTopK];
};

struct FrameParams {
  // configuration
  int L, H, NH, NKV, D, F, P, V, C0V, K, top_k, qk_norm, wdtype, draft_mode;
  float eps, T, sigma;
  unsigned long long seed;
  // geometry
  MatGeom g[MAT_COUNT];
  int qkv_dim;                 // NH*D + 2*NKV*D
  // weights
  const uint8_t* w_qkv;        // + l * g[MAT_QKV].stride
  const uint8_t* w_wo;
  const uint8_t* w_gu;
  const uint8_t* w_wd;
  const uint8_t* w_head;       // + (P-1) * g[MAT_HEAD].stride
  // W8A16: per tiled output row scales (null otherwise)
  const float* s_qkv;          // [L][qkv_dim]
  const float* s_wo;           // [L][H]
  const float* s_gu;           // [L][2F], tiled row order (gate rows 16t..16t+7, up rows +8)
  const float* s_wd;           // [L][H]
  const float* s_head;         // [n_pos][V]
  const float* attn_norm;      // [L][H]
  const float* ffn_norm;       // [L][H]
  const float* q_norm;         // [L][D]
  const float* k_norm;         // [L][D]
  const float* final_norm;     // [H]
  const float* offsets;        // [K][H]
  const float* head_bias;      // [n_pos][K][V]: LMH_P b_j, the offsets' share of the draft logits
  const uint8_t* embed;        // table i at embed + i * embed_stride (row-major, weight dtype)
  long long embed_stride;
  const float2* rope;          // [kMaxPos][D/2] (cos, sin)
  // buffers
  float* x;                    // [kMaxCols][H]
  float* qkv;                  // [kMaxCols][qkv_dim]
  float* mbuf;                 // [kMaxCols][F]
  float* attn;                 // [kMaxCols][NH*D] attention outputs (batched calls)
  float* logits;               // [kMaxTreeRows][kMaxDraft+1][V] (rows of one call)
  float* kcache;               // [S][L][NKV][kv_slots][D]
  float* vcache;
  TopkRec* topk;               // [2][kMaxCols][kMaxDraft+1]; a tree call: [kMaxTreeRows][kMaxDraft+1]
  TopkRec* draftq;             // [kMaxDraft] pending drafts' q
  DevState* st;                // [S]
  unsigned* ctr;               // [kMaxCalls][ctr_stride]
  int ctr_stride;
  int* err;                    // context-wide error word
  uint8_t* trace;              // optional
  // frame inputs
  const float* cond;           // [S][H]
  const int* c0;               // [S]
  const float* c0emb;          // [S][H]
  int S;                       // streams of this launch
  unsigned stream_ids[kMaxStreams], frame_ids[kMaxStreams];
  int* codes_out;              // [S][n_pos]
  mcd_frame_stats* stats;      // [S]
  long long kv_stride;         // floats between streams' KV caches
  int kv_slots;                // cache entries per (layer, KV head): positions 0..kMaxPos-1, then
                               // (TREE mode) the current tree call's rows at kMaxPos + row
  long long trace_stride;      // bytes between streams' trace blocks
  float* logits_out;           // stepwise: verify logits of the single call
  int* emitted_out;
  int* n_emitted_out;
  unsigned long long* timeline;  // optional [kMaxCalls][32] %globaltimer stamps (CTA 0)
  int single_call;             // 1 = run exactly one call (stepwise API)
  // sparse tree (TREE mode): nodes in breadth-first order
  int tree_n, tree_maxd;
  signed char tree_parent[kMaxTree], tree_rank[kMaxTree], tree_depth[kMaxTree];
  int tree_m[kMaxDraft];       // candidates needed per depth
  unsigned long long tree_anc[kMaxTree];   // node i: bit j set iff node j is i or an ancestor of i
  int* tree_cand;              // [kMaxDraft][kMaxTreeRank] candidates of the next call
  int n_cta;
  unsigned long long wait_ns;  // bound of every device-side wait
};

// Counter slots of one call (per layer 4 stages, then heads, top-k, call ready).
__host__ __device__ inline int ctr_stage(int layer, int s) { return layer * 4 + s; }
__host__ __device__ inline int ctr_heads(int L) { return L * 4; }
__host__ __device__ inline int ctr_topk(int L) { return L * 4 + 1; }
__host__ __device__ inline int ctr_ready(int L) { return L * 4 + 2; }
__host__ __device__ inline int ctr_accept(int L) { return L * 4 + 3; }
__host__ __device__ inline int ctr_att(int L, int layer) { return L * 4 + 4 + layer; }   // batched attention
__host__ __device__ inline int ctr_count(int L) { return L * 5 + 4; }

// ---------------------------------------------------------------------------------------
// PTX helpers
// ---------------------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }

// 1-D bulk copy global -> shared, completion counted on `bar` (16-B aligned, size % 16 == 0).
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar,
                                         uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar)), "l"(policy)
      : "memory");
}
__device__ __forceinline__ uint64_t policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint32_t ld_acquire(const unsigned* p) {
  uint32_t v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}
// Release-ordered add at GPU scope: every write that precedes it in this thread, or in the
// CTA's threads before a CTA barrier this thread passed, is visible to a thread that reads
// the new value with an acquire load.
__device__ __forceinline__ void red_release_add(unsigned* p, unsigned v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
// Acquire-release add at GPU scope returning the old value: releases like red_release_add
// and, for the caller (and its CTA after a barrier), acquires every write released by the
// earlier adds to the same counter.
__device__ __forceinline__ unsigned atom_add_acq_rel(unsigned* p, unsigned v) {
  unsigned old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
  return old;
}
// 16-byte global -> shared copy through L2 (cp.async.cg: other CTAs' writes are seen once
// they are visible at GPU scope); cpa_wait_all waits for this thread's copies.
__device__ __forceinline__ void cpa16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cpa_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }
// fp32 add of four consecutive words (16-byte aligned) at GPU scope as one vector reduction:
// a quarter of the L2 atomic operations of four scalar adds.
__device__ __forceinline__ void red_add_f32x4(float* p, float4 v) {
  asm volatile("red.global.add.v4.f32 [%0], {%1, %2, %3, %4};" ::"l"(p), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w)
               : "memory");
}
__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void consumer_sync() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint4& a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};\n"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a.x), "r"(a.y), "r"(a.z), "r"(a.w), "r"(b0), "r"(b1));
}

// fp32 -> (hi, lo) bf16 pair with x ~= hi + lo (round-to-nearest-even on both).
__device__ __forceinline__ uint32_t bf16_rn_bits(float x) {
  uint32_t u = __float_as_uint(x);
  uint32_t bias = ((u >> 16) & 1u) + 0x7FFFu;
  return (u + bias) >> 16;
}
__device__ __forceinline__ float bf16_bits_to_f32(uint32_t b) { return __uint_as_float(b << 16); }
// Two fp32 values rounded to nearest-even bf16 in one packed word: `lo` in bits 0-15.
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}
__device__ __forceinline__ float bf16_lo_f32(uint32_t w) { return __uint_as_float(w << 16); }
// Output-row scale of a W8A16 matrix (1 for 16- and 32-bit weights).
template <int WT>
__device__ __forceinline__ float wscale(const float* s, size_t i) {
  if (WT == MCD_WEIGHT_INT8) return __ldg(s + i);
  return 1.f;
}

// Eight signed bytes (an A fragment of a W8A16 tile) as eight bf16 values, exactly
// (|q| <= 127 needs 7 mantissa bits): bytes 2i, 2i+1 -> bf16 pair i (low half first).
__device__ __forceinline__ uint4 widen_i8x8(uint2 q) {
  auto pair = [](uint32_t w, int sh) {
    const float lo = (float)(int)(signed char)(w >> sh), hi = (float)(int)(signed char)(w >> (sh + 8));
    uint32_t d;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
    return d;
  };
  return make_uint4(pair(q.x, 0), pair(q.x, 16), pair(q.y, 0), pair(q.y, 16));
}
__device__ __forceinline__ float bf16_hi_f32(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ void split_bf16(float x, uint32_t& hi, uint32_t& lo) {
  hi = bf16_rn_bits(x);
  lo = bf16_rn_bits(x - bf16_bits_to_f32(hi));
}

// ---------------------------------------------------------------------------------------
// Philox4x32-10 (Salmon et al., SC'11) and the counter contract of mcd.h
// ---------------------------------------------------------------------------------------
__host__ __device__ inline void philox4x32_10(uint32_t c[4], uint32_t k0, uint32_t k1) {
  const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u, W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;
  for (int r = 0; r < 10; ++r) {
    if (r) {
      k0 += W0;
      k1 += W1;
    }
    uint64_t p0 = (uint64_t)M0 * c[0];
    uint64_t p1 = (uint64_t)M1 * c[2];
    uint32_t n0 = (uint32_t)(p1 >> 32) ^ c[1] ^ k0;
    uint32_t n2 = (uint32_t)(p0 >> 32) ^ c[3] ^ k1;
    c[0] = n0;
    c[1] = (uint32_t)p1;
    c[2] = n2;
    c[3] = (uint32_t)p0;
  }
}
__host__ __device__ inline double res53(uint32_t w0, uint32_t w1) {
  return ((double)(w0 >> 5) * 67108864.0 + (double)(w1 >> 6)) * (1.0 / 9007199254740992.0);
}
__host__ __device__ inline void philox_block(unsigned long long seed, uint32_t stream, uint32_t frame, int call,
                                             int pos, uint32_t purpose, uint32_t out[4]) {
  out[0] = stream;
  out[1] = frame;
  out[2] = ((uint32_t)call << 8) | (uint32_t)pos;
  out[3] = purpose;
  philox4x32_10(out, (uint32_t)(seed & 0xFFFFFFFFull), (uint32_t)(seed >> 32));
}
// The 53-bit integer uniform of a decision: u = U / 2^53 = res53(w0, w1).  (Not inlined on
// the device: the acceptance step draws several, and one copy of the rounds is enough.)
__host__ __device__ inline __noinline__ unsigned long long uniform_U(unsigned long long seed, uint32_t stream, uint32_t frame,
                                                        int call, int pos, uint32_t purpose) {
  uint32_t w[4];
  philox_block(seed, stream, frame, call, pos, purpose, w);
  return ((unsigned long long)(w[0] >> 5) << 26) | (unsigned long long)(w[1] >> 6);
}

enum { PURPOSE_TARGET = 0, PURPOSE_ACCEPT = 1, PURPOSE_DRAFT = 2, PURPOSE_NOISE = 3 };
constexpr uint32_t kPurposeSibling = 0x10000u;   // + i: test i >= 1 at a tree node

// Two N(0,1) draws for vocabulary entries (2 pair, 2 pair + 1) of a noisy draft row: the
// Box-Muller transform (Box and Muller, 1958) of the 53-bit uniforms of words (0,1) and
// (2,3) of purpose 3 + pair, radius sqrt(-2 ln(1 - u1)), angle 2 pi u2, in fp64.
__device__ inline __noinline__ double2 normal_pair(unsigned long long seed, uint32_t stream, uint32_t frame, int round,
                                      int position, int pair) {
  uint32_t c[4] = {stream, frame, ((uint32_t)round << 8) | (uint32_t)position, (uint32_t)(PURPOSE_NOISE + pair)};
  philox4x32_10(c, (uint32_t)seed, (uint32_t)(seed >> 32));
  const double u1 = ((double)(c[0] >> 5) * 67108864.0 + (double)(c[1] >> 6)) * (1.0 / 9007199254740992.0);
  const double u2 = ((double)(c[2] >> 5) * 67108864.0 + (double)(c[3] >> 6)) * (1.0 / 9007199254740992.0);
  const double r = sqrt(-2.0 * log(1.0 - u1));
  const double t = 2.0 * 3.141592653589793 * u2;
  double sn, cs;
  sincos(t, &sn, &cs);
  return make_double2(r * cs, r * sn);
}

// ---------------------------------------------------------------------------------------
// Bounded waits: every spin gives up after wait_ns and records MCD_ERR_TIMEOUT.
// ---------------------------------------------------------------------------------------
__device__ __forceinline__ bool wait_counter(const unsigned* p, unsigned target, int* err,
                                             unsigned long long wait_ns) {
  if (ld_acquire(p) >= target) return true;
  uint64_t t0 = globaltimer();
  uint32_t it = 0;
  while (ld_acquire(p) < target) {
    if ((++it & 63u) == 0) {
      if (*(volatile int*)err != 0) return false;
      if (globaltimer() - t0 > wait_ns) {
        atomicCAS(err, 0, (int)MCD_ERR_TIMEOUT);
        return false;
      }
    }
  }
  return true;
}

__device__ __forceinline__ bool wait_mbar(uint64_t* bar, uint32_t parity, int* err, unsigned long long wait_ns,
                                          const volatile int* stop) {
  if (mbar_try_wait(bar, parity)) return true;
  uint64_t t0 = globaltimer();
  uint32_t it = 0;
  while (!mbar_try_wait(bar, parity)) {
    if ((++it & 15u) == 0) {
      if (stop && *stop) return false;
      if (*(volatile int*)err != 0) return false;
      if (globaltimer() - t0 > wait_ns) {
        atomicCAS(err, 0, (int)MCD_ERR_TIMEOUT);
        return false;
      }
    }
  }
  return true;
}

}  // namespace mcd
