// Outer CodeDecoder and the full frame pipeline (arXiv 2609.37007, Sec. 1 and Fig. 1).
//
// Per 80 ms frame the CodeDecoder (28 pre-norm layers, the MultiCodeDecoder's block) runs
// one row over its utterance-long KV cache, its c0 head gives the frame's seed code c0 (top-k
// / temperature sampling, Philox counter of position 0), and its post-norm hidden state plus
// the c0 embedding start the MultiCodeDecoder's frame, which emits c1..c15.  The next
// frame's CodeDecoder input is the sum of the text row (if any) and the embeddings of the 16
// codes just emitted.  Before frame 0 the text prompt is prefilled: with the shapes the
// tcgen05 block kernels take, all rows but the last as one batch on the tensor cores
// (outer_tc_prefill), else up to 16 rows per outer_kernel launch; the last row always runs
// through outer_kernel, which samples frame 0's c0.
//
// outer_kernel is one cooperative launch of one CTA per SM, built on the same weight ring
// and unit GEMMs as the frame kernel (mcd_stage.cuh): per layer QKV -> attention -> Wo ->
// gate/up -> down, each stage ordered by a grid-wide arrival counter.  Attention over the
// long cache is split over key blocks (flash-decoding style): one task per (KV head, block
// of 32 keys) normalises and rotates its rows' queries and new keys, writes the new K / V
// to the cache (rounded to the cache dtype), and leaves per-row partial softmax sums
// (max, sum of exponentials, weighted values); the CTAs of the Wo stage merge the blocks of
// their head before multiplying.  The last CTA to finish the c0 head samples c0.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <map>
#include <string>
#include <vector>

#include "../../include/mcd_pipeline.h"
#include "mcd_host.cuh"
#include "mcd_internal.cuh"
#include "mcd_sampler.cuh"
#include "mcd_stage.cuh"
#include "mcd_tcops.cuh"

namespace mcd {

constexpr int kKeyBlock = 32;          // keys per attention task
constexpr int kMaxOuterTokens = 1024;  // KV capacity: at most 32 key blocks (one lane each)
constexpr int kMaxPrefillRows = 16;    // rows per prefill launch (bf16 hi/lo operand)
constexpr int kMaxQVec = 32;           // query vectors per attention task (rows x group)
constexpr int kPartLd = 132;           // floats per partial record: D (<= 128) values, max, sum

struct OuterStep {
  uint8_t* kcache;                 // [L][NKV][cap][D] in the weight dtype
  uint8_t* vcache;
  int cap;
  const float2* rope;              // [cap][D/2] (cos, sin)
  int pos0, nr, head;              // first new position, new rows, 1 = c0 head + sampling
  const int* text_ids;             // prefill: ids of the rows (device), else null
  const int* prev_codes;           // frame step: c0..c_P of the previous frame (device)
  int text_id;                     // frame step: text row added to the sum, -1 = none
  const uint8_t* text_table;
  int text_vocab;
  const uint8_t* c0_table;
  int c0_vocab;
  const uint8_t* code_tables;      // inner table j (1 <= j < P) at code_tables + j * code_stride
  long long code_stride;
  int code_vocab, P;
  const uint8_t* last_table;       // table P (owned by the outer model)
  float* part;                     // [n_blocks][nr][NH][kPartLd]
  int* c0_out;
  int* c0_out2;                    // optional second destination of c0
  float* cond_out;                 // [H] post-norm hidden state of the last row
  float* c0emb_out;                // [H] c0 embedding (fp32)
  float* trace;                    // optional [C0V + 2H]: c0 logits, cond, c0 embedding
  unsigned stream_id, frame_id;
};

// ------------------------------------------------------------------------------------
// Producer: the CTA's units of every stage, in stage order.
// ------------------------------------------------------------------------------------
__device__ void outer_producer(const FrameParams& p, const OuterStep& o, Smem& sm) {
  const uint64_t pol = policy_evict_first();
  const volatile int* stop = sm.flags;
  const int heads[1] = {1};
  const int ns = 4 * p.L + (o.head ? 1 : 0);
  uint32_t issued = 0;
  int rot = 0;
  bool halt = false;
  for (int si = 0; si < ns && !halt; ++si) {
    const int n = stage_units(p, si, 1);
    const uint32_t bytes = (uint32_t)p.g[stage_kind(si, p.L)].unit_bytes;
    const UnitRange ur = unit_range(si, p.L, n, blockIdx.x, rot, p.n_cta);
    for (int u = ur.first; u < ur.end && !halt; u += ur.step)
      halt = !ring_issue(p, sm, issued, unit_src(p, si, u, heads), bytes, pol, stop);
    rot = (rot + n) % p.n_cta;
  }
  ring_drain(p, sm, issued);
}

// ------------------------------------------------------------------------------------
// Attention task (KV head g, key block b)
// ------------------------------------------------------------------------------------
// Keys j0..j1-1 of the block: cached positions (< pos0) come from the cache, new positions
// from this launch's QKV output.  Query vector qi is row n_lo + qi / group, query head
// g * group + qi % group; rows below n_lo see no key of the block.  Scratch (act + bfrag):
// q [32][D + 8], k [32][D + 8], v [32][D], scores [32][32], rope rows [16][D/2], gains.
template <int WT>
__device__ void outer_attention(Cons& c, const OuterStep& o, int layer, int g, int b) {
  const FrameParams& p = c.p;
  const int D = p.D, half = D >> 1, group = p.NH / p.NKV, nr = o.nr, pos0 = o.pos0;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int j0 = b * kKeyBlock, j1 = min(j0 + kKeyBlock, pos0 + nr), nk = j1 - j0;
  const int jn = min(max(j0, pos0), j1);      // first new key of the block (j1: none)
  const int n_lo = max(0, j0 - pos0);         // first row that sees a key of the block
  const int nq = (nr - n_lo) * group;
  const int KS = D + 8;
  const int cpr = D >> 2;                     // 16-byte fp32 chunks per row
  float* qs = c.sm.act;
  float* ks = qs + kMaxQVec * 136;
  float* vs = ks + kKeyBlock * 136;
  float* sc = vs + kKeyBlock * 128;
  float2* cs = reinterpret_cast<float2*>(sc + kMaxQVec * kKeyBlock);
  float* gq = reinterpret_cast<float*>(cs + kMaxPrefillRows * 64);
  float* gk = gq + 128;
  const size_t es = WT == MCD_WEIGHT_BF16 ? 2 : 4;
  const size_t cache_off = (((size_t)layer * p.NKV + g) * o.cap) * D;   // elements
  const int qkv_dim = p.qkv_dim, koff = p.NH * D + g * D, voff = p.NH * D + p.NKV * D + g * D;
  // ---- (A) loads, 16-byte chunks, a batch of 8 per thread in flight -----------------------
  {
    const int e_q = nq * cpr;                         // queries
    const int e_new = e_q + 2 * (j1 - jn) * cpr;      // new keys then new values
    const int ccpr = WT == MCD_WEIGHT_BF16 ? (D >> 3) : cpr;   // chunks per cached row
    const int e_old = e_new + 2 * (jn - j0) * ccpr;   // cached keys then cached values
    const int e_cs = e_old + (nr - n_lo) * (half >> 1);
    const int e_all = e_cs + (p.qk_norm ? 2 * cpr : 0);
    for (int base = 0; base < e_all; base += 8 * kConsumerThreads) {
      float4 v[8];
      int kind[8];
      void* dst[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int i = base + tid + u * kConsumerThreads;
        kind[u] = -1;
        if (i >= e_all) continue;
        if (i < e_q) {
          const int qi = i / cpr, ch = i - qi * cpr, n = n_lo + qi / group, h = g * group + qi % group;
          v[u] = __ldcg(reinterpret_cast<const float4*>(p.qkv + (size_t)n * qkv_dim + h * D) + ch);
          dst[u] = reinterpret_cast<float4*>(qs + qi * KS) + ch;
          kind[u] = 0;
        } else if (i < e_new) {
          const int r = i - e_q, isv = r >= (j1 - jn) * cpr, rr = r - (isv ? (j1 - jn) * cpr : 0);
          const int jj = rr / cpr, ch = rr - jj * cpr, n = jn + jj - pos0;
          v[u] = __ldcg(reinterpret_cast<const float4*>(p.qkv + (size_t)n * qkv_dim + (isv ? voff : koff)) + ch);
          dst[u] = isv ? reinterpret_cast<float4*>(vs + (jn + jj - j0) * D) + ch
                       : reinterpret_cast<float4*>(ks + (jn + jj - j0) * KS) + ch;
          kind[u] = 0;
        } else if (i < e_old) {
          const int r = i - e_new, isv = r >= (jn - j0) * ccpr, rr = r - (isv ? (jn - j0) * ccpr : 0);
          const int jj = rr / ccpr, ch = rr - jj * ccpr;
          const uint8_t* src = (isv ? o.vcache : o.kcache) + (cache_off + (size_t)(j0 + jj) * D) * es;
          v[u] = __ldcg(reinterpret_cast<const float4*>(src) + ch);
          float* row = isv ? vs + jj * D : ks + jj * KS;
          dst[u] = row + ch * (WT == MCD_WEIGHT_BF16 ? 8 : 4);
          kind[u] = WT == MCD_WEIGHT_BF16 ? 1 : 0;
        } else if (i < e_cs) {
          const int r = i - e_old, n = n_lo + r / (half >> 1), ch = r % (half >> 1);
          v[u] = __ldg(reinterpret_cast<const float4*>(o.rope + (size_t)(pos0 + n) * half) + ch);
          dst[u] = reinterpret_cast<float4*>(cs + n * 64) + ch;
          kind[u] = 0;
        } else {
          const int r = i - e_cs, w = r / cpr, ch = r - w * cpr;
          v[u] = __ldg(reinterpret_cast<const float4*>((w == 0 ? p.q_norm : p.k_norm) + (size_t)layer * D) + ch);
          dst[u] = reinterpret_cast<float4*>(w == 0 ? gq : gk) + ch;
          kind[u] = 0;
        }
      }
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        if (kind[u] == 0) {
          *reinterpret_cast<float4*>(dst[u]) = v[u];
        } else if (kind[u] == 1) {   // 8 bf16 -> 8 floats
          const uint32_t w[4] = {__float_as_uint(v[u].x), __float_as_uint(v[u].y), __float_as_uint(v[u].z),
                                 __float_as_uint(v[u].w)};
          float4* d4 = reinterpret_cast<float4*>(dst[u]);
          d4[0] = make_float4(bf16_lo_f32(w[0]), bf16_hi_f32(w[0]), bf16_lo_f32(w[1]), bf16_hi_f32(w[1]));
          d4[1] = make_float4(bf16_lo_f32(w[2]), bf16_hi_f32(w[2]), bf16_lo_f32(w[3]), bf16_hi_f32(w[3]));
        }
      }
    }
  }
  consumer_sync();
  // ---- (B) QK-norm + RoPE of the queries and new keys; new K / V rounded and cached -------
  const int nd = D >> 5;   // dims per lane (lane + 32 i)
  const int n_new = j1 - jn;
  for (int vi = warp; vi < nq + 2 * n_new; vi += kConsumerWarps) {
    const int kind = vi < nq ? 0 : (vi < nq + n_new ? 1 : 2);   // query, new key, new value
    const int jj = kind == 0 ? 0 : (kind == 1 ? vi - nq : vi - nq - n_new);
    const int n = kind == 0 ? n_lo + vi / group : jn + jj - pos0;
    float* row = kind == 0 ? qs + vi * KS : (kind == 1 ? ks + (jn + jj - j0) * KS : vs + (jn + jj - j0) * D);
    float x[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) x[i] = i < nd ? row[lane + 32 * i] : 0.f;
    if (kind < 2) {
      if (p.qk_norm) {
        float ss = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i) ss += x[i] * x[i];
#pragma unroll
        for (int off = 16; off; off >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, off);
        const float scl = rsqrtf(ss / (float)D + p.eps);
        const float* gg = kind == 0 ? gq : gk;
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (i < nd) x[i] = x[i] * scl * gg[lane + 32 * i];
      }
#pragma unroll
      for (int i = 0; i < 2; ++i) {
        if (i < nd / 2) {
          const float2 r = cs[n * 64 + lane + 32 * i];
          const float a = x[i], bb = x[i + nd / 2];
          x[i] = a * r.x - bb * r.y;
          x[i + nd / 2] = bb * r.x + a * r.y;
        }
      }
    }
    if (kind > 0) {   // cache dtype: the value every later read sees, this task's included
      uint8_t* dst = (kind == 1 ? o.kcache : o.vcache) + (cache_off + (size_t)(pos0 + n) * D) * es;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        if (i < nd) {
          if (WT == MCD_WEIGHT_BF16) {
            const uint32_t bits = bf16_rn_bits(x[i]);
            reinterpret_cast<uint16_t*>(dst)[lane + 32 * i] = (uint16_t)bits;
            x[i] = bf16_bits_to_f32(bits);
          } else {
            reinterpret_cast<float*>(dst)[lane + 32 * i] = x[i];
          }
        }
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (i < nd) row[lane + 32 * i] = x[i];
  }
  consumer_sync();
  // ---- (C) scores: two threads per (query, key), interleaved 16-byte chunks ---------------
  const float scale = rsqrtf((float)D);
  for (int t = tid; t < nq * 2 * kKeyBlock; t += kConsumerThreads) {
    const int qi = t / (2 * kKeyBlock), kk = (t >> 1) & (kKeyBlock - 1), hf = t & 1;
    const int n = n_lo + qi / group;
    const bool live = kk < nk && j0 + kk <= pos0 + n;
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
    if (live) {
      const float4* q4 = reinterpret_cast<const float4*>(qs + qi * KS) + hf;
      const float4* k4 = reinterpret_cast<const float4*>(ks + kk * KS) + hf;
#pragma unroll 8
      for (int ch = 0; ch < (cpr >> 1); ++ch) {
        const float4 q = q4[2 * ch], k = k4[2 * ch];
        a0 += q.x * k.x;
        a1 += q.y * k.y;
        a2 += q.z * k.z;
        a3 += q.w * k.w;
      }
    }
    float acc = (a0 + a1) + (a2 + a3);
    acc += __shfl_xor_sync(0xFFFFFFFFu, acc, 1);
    if (hf == 0) sc[qi * kKeyBlock + kk] = live ? acc * scale : -INFINITY;
  }
  consumer_sync();
  // ---- (D) block softmax statistics: one warp per query (lane = key) ------------------------
  for (int qi = warp; qi < nq; qi += kConsumerWarps) {
    const int n = n_lo + qi / group, h = g * group + qi % group;
    const float s = sc[qi * kKeyBlock + lane];
    float m = s;
#pragma unroll
    for (int off = 16; off; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, off));
    const float e = s == -INFINITY ? 0.f : __expf(s - m);
    float l = e;
#pragma unroll
    for (int off = 16; off; off >>= 1) l += __shfl_xor_sync(0xFFFFFFFFu, l, off);
    sc[qi * kKeyBlock + lane] = e;
    if (lane == 0) {
      float* rec = o.part + (((size_t)b * nr + n) * p.NH + h) * kPartLd;
      rec[D] = m;
      rec[D + 1] = l;
    }
  }
  consumer_sync();
  // ---- (E) weighted values: one thread per (query, dim pair) -------------------------------
  for (int t = tid; t < nq * half; t += kConsumerThreads) {
    const int qi = t / half, d = 2 * (t - qi * half);
    const int n = n_lo + qi / group, h = g * group + qi % group;
    const float* pr = sc + qi * kKeyBlock;
    float2 acc = make_float2(0.f, 0.f);
    for (int kk = 0; kk < nk; ++kk) {
      const float w = pr[kk];
      const float2 v = *reinterpret_cast<const float2*>(vs + kk * D + d);
      acc.x += w * v.x;
      acc.y += w * v.y;
    }
    *reinterpret_cast<float2*>(o.part + (((size_t)b * nr + n) * p.NH + h) * kPartLd + d) = acc;
  }
  consumer_sync();
}

// Attention output of query head h for every row: the merge of the key blocks' partial sums
// (each block rescaled by e^{m_b - M}), written to ao [nr][D] in shared memory.
__device__ void outer_merge(Cons& c, const OuterStep& o, int h, float* ao) {
  const FrameParams& p = c.p;
  const int D = p.D, nr = o.nr, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  float* wts = ao + kMaxPrefillRows * 128;     // [nr][32] block weights / denominator
  for (int n = warp; n < nr; n += kConsumerWarps) {
    const int nb = (o.pos0 + n) / kKeyBlock + 1;
    float m = -INFINITY, l = 0.f;
    if (lane < nb) {
      const float* rec = o.part + (((size_t)lane * nr + n) * p.NH + h) * kPartLd;
      m = __ldcg(rec + D);
      l = __ldcg(rec + D + 1);
    }
    float M = m;
#pragma unroll
    for (int off = 16; off; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xFFFFFFFFu, M, off));
    const float w = lane < nb ? __expf(m - M) : 0.f;
    float den = w * l;
#pragma unroll
    for (int off = 16; off; off >>= 1) den += __shfl_xor_sync(0xFFFFFFFFu, den, off);
    wts[n * 32 + lane] = w / den;
  }
  consumer_sync();
  for (int i = tid; i < nr * D; i += kConsumerThreads) {
    const int n = i / D, d = i - n * D, nb = (o.pos0 + n) / kKeyBlock + 1;
    float acc = 0.f;
    for (int b = 0; b < nb; ++b)
      acc += wts[n * 32 + b] * __ldcg(o.part + (((size_t)b * nr + n) * p.NH + h) * kPartLd + d);
    ao[n * D + d] = acc;
  }
  consumer_sync();
}

// c0 of the frame (run by the CTA that finished the c0 head last): top-k / temperature
// distribution of the logits, one draw with counter (stream, frame, 0, 0, 0); then the
// inner model's inputs: cond = post-norm hidden state, the c0 embedding in fp32.
template <int WT>
__device__ void outer_sample(Cons& c, const OuterStep& o) {
  const FrameParams& p = c.p;
  Smem& sm = c.sm;
  TopkScratch& ts = *reinterpret_cast<TopkScratch*>(sm.act);
  TopkRec* rec = reinterpret_cast<TopkRec*>(sm.bfrag);
  __shared__ int s_c0;
  block_topk(p.logits, p.V, p.top_k, p.T, 0, ts, rec);
  consumer_sync();
  if (threadIdx.x < 32) {
    const unsigned long long U = uniform_U(p.seed, o.stream_id, o.frame_id, 0, 0, PURPOSE_TARGET);
    const int d = warp_draw(rec, U);
    if (threadIdx.x == 0) s_c0 = d;
  }
  consumer_sync();
  const int c0 = s_c0;
  if (threadIdx.x == 0) {
    *o.c0_out = c0;
    if (o.c0_out2) *o.c0_out2 = c0;
  }
  const float inv = sm.inv_rms[0];
  const float* xl = p.x + (size_t)(o.nr - 1) * p.H;
  for (int k = threadIdx.x; k < p.H; k += kConsumerThreads) {
    const float h = __ldcg(xl + k) * inv * sm.vec[k];
    const float e = WT == MCD_WEIGHT_BF16
                        ? bf16_bits_to_f32(reinterpret_cast<const uint16_t*>(o.c0_table)[(size_t)c0 * p.H + k])
                        : reinterpret_cast<const float*>(o.c0_table)[(size_t)c0 * p.H + k];
    o.cond_out[k] = h;
    o.c0emb_out[k] = e;
    if (o.trace) {
      o.trace[p.V + k] = h;
      o.trace[p.V + p.H + k] = e;
    }
  }
  if (o.trace)
    for (int i = threadIdx.x; i < p.V; i += kConsumerThreads) o.trace[i] = __ldcg(p.logits + i);
}

// ------------------------------------------------------------------------------------
// One launch: prefill rows or one frame row
// ------------------------------------------------------------------------------------
template <int WT, bool WIDE>
__device__ void run_outer(Cons& c, const OuterStep& o) {
  const FrameParams& p = c.p;
  Smem& sm = c.sm;
  const int L = p.L, H = p.H, D = p.D, F = p.F, nr = o.nr;
  unsigned* ctr = p.ctr;
  const unsigned N = (unsigned)p.n_cta;
  const size_t rb = (size_t)H * (WT == MCD_WEIGHT_BF16 ? 2 : 4);   // bytes per table row
  int* ids = sm.ci->r_id;    // prefill: text id per row; frame: c0..c_P, then the text id
  if (threadIdx.x < kMaxCols) {
    const int t = threadIdx.x;
    int id = -1, lim = 0;
    if (o.text_ids) {
      if (t < nr) {
        id = o.text_ids[t];
        lim = o.text_vocab;
      }
    } else if (t <= o.P) {
      id = o.prev_codes[t];
      lim = t == 0 ? o.c0_vocab : o.code_vocab;
    } else if (t == o.P + 1 && o.text_id >= 0) {
      id = o.text_id;
      lim = o.text_vocab;
    }
    if (lim > 0 && (id < 0 || id >= lim)) {   // an id outside its table: fail the step
      atomicCAS(p.err, 0, (int)MCD_ERR_INVALID_ARG);
      id = 0;
    }
    ids[t] = id;
  }
  // layer-0 row n: a prompt row, or the frame input text + E_c0(c0) + sum_j E_j(c_j)
  auto ld0 = [&](int n, int k, auto w) {
    constexpr int W = decltype(w)::value;
    auto row_v = [&](const uint8_t* row) {
      if constexpr (WT == MCD_WEIGHT_BF16) return ldg_bf16_v<W>(row, k);
      else return ldg_f32_v<W>(row, k);
    };
    if (o.text_ids) return row_v(o.text_table + (size_t)ids[n] * rb);
    vecf<W> s{};
    if (ids[o.P + 1] >= 0) s = row_v(o.text_table + (size_t)ids[o.P + 1] * rb);
    add_v<W>(s, row_v(o.c0_table + (size_t)ids[0] * rb));
    for (int j = 1; j < o.P; ++j) add_v<W>(s, row_v(o.code_tables + (long long)j * o.code_stride + (size_t)ids[j] * rb));
    add_v<W>(s, row_v(o.last_table + (size_t)ids[o.P] * rb));
    return s;
  };
  auto from_x = [&](int n, int k, auto w) { return ld_global_v<decltype(w)::value>(p.x + (size_t)n * H + k); };
  auto no_key = [](int) { return 0; };
  auto no_prep = [](int, int, int) {};
  const int n_blocks = (o.pos0 + nr + kKeyBlock - 1) / kKeyBlock;

  for (int l = 0; l < L; ++l) {
    // ---- RMSNorm -> QKV -----------------------------------------------------------------
    g2s_vec(sm.vec, p.attn_norm + (size_t)l * H, H);
    if (l == 0) {
      consumer_sync();                       // gain and ids in shared memory
      prep_operand<WT, WIDE>(c, nr, H, 0, H, sm.vec, true, ld0, blockIdx.x == 0 ? p.x : nullptr);
    } else {
      if (!cons_wait(c, ctr + ctr_stage(l - 1, 3), N)) return;
      prep_operand<WT, WIDE>(c, nr, H, 0, H, sm.vec, true, from_x);
    }
    {
      const MatGeom& g = p.g[MAT_QKV];
      run_stage<WT, WIDE>(c, 0, 4 * l + 0, g.n_units, H, nr, no_key, no_prep,
                          [&](int u, int mi, int rr, int n, float v, float) {
                            const int row = (u % g.n_mb) * g.Mu * 16 + mi * 16 + rr;
                            p.qkv[(size_t)n * p.qkv_dim + row] = v * sm.inv_rms[n];
                          });
      if (c.abort_) return;
    }
    cons_signal(c, ctr + ctr_stage(l, 0), 0, 0);

    // ---- attention: (KV head, key block) tasks, then one grid barrier -------------------------
    if (!cons_wait(c, ctr + ctr_stage(l, 0), N)) return;
    for (int t = blockIdx.x; t < p.NKV * n_blocks; t += p.n_cta) outer_attention<WT>(c, o, l, t % p.NKV, t / p.NKV);
    cons_signal(c, ctr + ctr_att(L, l), 0, 0);
    if (!cons_wait(c, ctr + ctr_att(L, l), N)) return;

    // ---- Wo + residual: unit u multiplies the merged output of head u / n_mb ----------------
    {
      const MatGeom& g = p.g[MAT_WO];
      float* ao = reinterpret_cast<float*>(sm.bfrag);
      if (threadIdx.x == 0) sm.flags[3] = -1;
      consumer_sync();
      run_stage<WT, WIDE>(
          c, 0, 4 * l + 1, g.n_units, D, nr, [&](int u) { return u / g.n_mb; },
          [&](int u, int, int) {
            const int h = u / g.n_mb;
            if (sm.flags[3] != h) {
              outer_merge(c, o, h, ao);
              prep_operand<WT, WIDE>(c, nr, D, 0, D, nullptr, false,
                                     [&](int n, int k, auto w) { return ld_shared_v<decltype(w)::value>(ao + n * D + k); });
              if (threadIdx.x == 0) sm.flags[3] = h;
            }
          },
          [&](int u, int mi, int rr, int n, float v, float) {
            const int row = (u % g.n_mb) * g.Mu * 16 + mi * 16 + rr;
            atomicAdd(p.x + (size_t)n * H + row, v);
          });
      if (c.abort_) return;
    }
    cons_signal(c, ctr + ctr_stage(l, 1), 0, 0);

    // ---- RMSNorm -> gate/up -> SwiGLU ---------------------------------------------------------
    g2s_vec(sm.vec, p.ffn_norm + (size_t)l * H, H);
    if (!cons_wait(c, ctr + ctr_stage(l, 1), N)) return;
    prep_operand<WT, WIDE>(c, nr, H, 0, H, sm.vec, true, from_x);
    {
      const MatGeom& g = p.g[MAT_GU];
      run_stage<WT, WIDE>(
          c, 0, 4 * l + 2, g.n_units, H, nr, no_key, no_prep,
          [&](int u, int mi, int rr, int n, float gate, float up) {
            const float s = sm.inv_rms[n];
            const float gt = gate * s;
            const int j = ((u % g.n_mb) * g.Mu + mi) * 8 + rr;
            p.mbuf[(size_t)n * F + j] = gt / (1.0f + __expf(-gt)) * (up * s);
          },
          true);
      if (c.abort_) return;
    }
    cons_signal(c, ctr + ctr_stage(l, 2), 0, 0);

    // ---- down + residual ------------------------------------------------------------------------
    if (!cons_wait(c, ctr + ctr_stage(l, 2), N)) return;
    {
      const MatGeom& g = p.g[MAT_WD];
      const int Kc = g.Ku * 16;
      if (threadIdx.x == 0) sm.flags[3] = -1;
      consumer_sync();
      run_stage<WT, WIDE>(
          c, 0, 4 * l + 3, g.n_units, Kc, nr, [&](int u) { return u / g.n_mb; },
          [&](int u, int, int) {
            const int kc = u / g.n_mb;
            if (sm.flags[3] != kc) {
              const float* m = p.mbuf + (size_t)kc * Kc;
              prep_operand<WT, WIDE>(c, nr, Kc, 0, Kc, nullptr, false,
                                     [&](int n, int k, auto w) { return ld_global_v<decltype(w)::value>(m + (size_t)n * F + k); });
              if (threadIdx.x == 0) sm.flags[3] = kc;
            }
          },
          [&](int u, int mi, int rr, int n, float v, float) {
            const int row = (u % g.n_mb) * g.Mu * 16 + mi * 16 + rr;
            atomicAdd(p.x + (size_t)n * H + row, v);
          });
      if (c.abort_) return;
    }
    cons_signal(c, ctr + ctr_stage(l, 3), 0, 0);
  }
  if (!o.head) return;

  // ---- final RMSNorm of the last row -> c0 head -------------------------------------------
  g2s_vec(sm.vec, p.final_norm, H);
  if (!cons_wait(c, ctr + ctr_stage(L - 1, 3), N)) return;
  const float* xl = p.x + (size_t)(nr - 1) * H;
  prep_operand<WT, WIDE>(c, 1, H, 0, H, sm.vec, true, [&](int, int k, auto w) { return ld_global_v<decltype(w)::value>(xl + k); });
  {
    const MatGeom& g = p.g[MAT_HEAD];
    run_stage<WT, WIDE>(c, 0, 4 * L, g.n_units, H, 1, no_key, no_prep,
                        [&](int u, int mi, int rr, int, float v, float) {
                          p.logits[(u % g.n_units) * g.Mu * 16 + mi * 16 + rr] = v * sm.inv_rms[0];
                        });
    if (c.abort_) return;
  }
  consumer_sync();
  if (threadIdx.x == 0) {
    __threadfence();
    const unsigned old = atomicAdd(ctr + ctr_heads(L), 1u);
    sm.flags[2] = old == N - 1u ? 1 : 0;
    if (sm.flags[2]) __threadfence();
  }
  consumer_sync();
  if (sm.flags[2]) outer_sample<WT>(c, o);
}

template <int WT, bool WIDE>
__global__ void __launch_bounds__(kThreads, 1)
    outer_kernel(const __grid_constant__ FrameParams p, const __grid_constant__ OuterStep o) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  Smem sm = smem_layout(smem_raw);
  const int tid = threadIdx.x, warp = tid >> 5;
  if (tid == 0) {
    for (int s = 0; s < kNumSlots; ++s) {
      mbar_init(&sm.full[s], 1);
      mbar_init(&sm.empty[s], kConsumerWarps);
    }
    sm.flags[0] = 0;
    sm.flags[1] = 0;
    sm.flags[2] = 0;
    sm.flags[3] = -1;
    fence_barrier_init();
  }
  __syncthreads();
  if (warp == kConsumerWarps) {
    if ((tid & 31) == 0) outer_producer(p, o, sm);
  } else {
    Cons c(p, sm);
    run_outer<WT, WIDE>(c, o);
    if (tid == 0) sm.flags[0] = 1;   // stop the producer
  }
  __syncthreads();
}

__global__ void outer_begin_kernel(unsigned* ctr, int n) {
  for (int i = threadIdx.x; i < n; i += blockDim.x) ctr[i] = 0u;
}

template <int WT, bool WIDE>
static void* outer_entry() {
  return (void*)outer_kernel<WT, WIDE>;
}

static void* outer_fn(int wdtype, bool wide) {
  return wdtype == MCD_WEIGHT_BF16 ? (wide ? outer_entry<MCD_WEIGHT_BF16, true>() : outer_entry<MCD_WEIGHT_BF16, false>())
                                   : (wide ? outer_entry<MCD_WEIGHT_F32, true>() : outer_entry<MCD_WEIGHT_F32, false>());
}

}  // namespace mcd

using namespace mcd;

// ------------------------------------------------------------------------------------
// Host side
// ------------------------------------------------------------------------------------
// Prompt prefill on the tensor cores: rows 0..T-2 of a T-token prompt go through the 28
// layers as one batch (tcgen05 products, causal attention, K / V written to the cache); the
// last row then runs through outer_kernel, which reads that cache and samples c0.
struct OuterTc {
  bool on = false;
  int Rtc = 0;                     // prompt rows, rounded up to the tile width
  uint8_t* w = nullptr;            // per layer: SW128 copies of the weights
  TcLayerOffsets off;
  float* X = nullptr;              // [Rtc][H] residual stream
  float* ss = nullptr;             // [Rtc] sums of squares (the next RMSNorm)
  float* qkv = nullptr;            // [Rtc][qkv_dim]
  float* q = nullptr;              // [Rtc][NH * D] normalised, rotated queries
  float* part = nullptr;           // [kTcSplit][Rtc][H] partial sums of the residual products
  uint8_t *xn_hi = nullptr, *xn_lo = nullptr, *att_t = nullptr, *act_t = nullptr;   // operands
  int* rows = nullptr;             // device: live rows
};

__global__ void pf_set_rows_kernel(int* rows, int n) { *rows = n; }

// Prompt rows: X = the rows' text embeddings (bf16 table), ss = their sums of squares.  One
// CTA per row, thread t owns elements 8t..8t+7.
__global__ void __launch_bounds__(128) pf_embed_kernel(const int* __restrict__ ids, const int* nrows,
                                                       const uint8_t* __restrict__ table, int vocab, int H, float* X,
                                                       float* ss, int* err) {
  const int r = blockIdx.x;
  if (r >= *nrows) return;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  int id = ids[r];
  if (id < 0 || id >= vocab) {              // an id outside the text table fails the prefill
    if (t == 0) atomicCAS(err, 0, (int)MCD_ERR_INVALID_ARG);
    id = 0;
  }
  __shared__ float red[4];
  float s2 = 0.f;
  if (t < H / 8) {
    const uint4 w = __ldg(reinterpret_cast<const uint4*>(table + ((size_t)id * H + 8 * t) * 2));
    const float v[8] = {bf16_lo_f32(w.x), bf16_hi_f32(w.x), bf16_lo_f32(w.y), bf16_hi_f32(w.y),
                        bf16_lo_f32(w.z), bf16_hi_f32(w.z), bf16_lo_f32(w.w), bf16_hi_f32(w.w)};
    float4* xr = reinterpret_cast<float4*>(X + (size_t)r * H + 8 * t);
    xr[0] = make_float4(v[0], v[1], v[2], v[3]);
    xr[1] = make_float4(v[4], v[5], v[6], v[7]);
#pragma unroll
    for (int i = 0; i < 8; ++i) s2 += v[i] * v[i];
  }
#pragma unroll
  for (int off = 16; off; off >>= 1) s2 += __shfl_xor_sync(0xFFFFFFFFu, s2, off);
  if (lane == 0) red[warp] = s2;
  __syncthreads();
  if (t == 0) ss[r] = red[0] + red[1] + red[2] + red[3];
}

// QK-norm + RoPE (position = row index) of every prompt row's query and key heads; K and V
// rounded to bf16 into layer l's cache ([NKV][cap][D]), the rotated queries (fp32) into q.
// One warp per (row, vector), lane holding dims lane + 32 i.
__global__ void __launch_bounds__(256) pf_rope_kv_kernel(const float* __restrict__ qkv, int qkv_dim, const int* nrows,
                                                         int NH, int NKV, int D, int qk_norm, const float* qn,
                                                         const float* kn, float eps, const float2* __restrict__ rope,
                                                         uint16_t* kc, uint16_t* vc, int cap, float* q) {
  const int vecs = NH + 2 * NKV, w = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  const int r = w / vecs, vi = w - r * vecs;
  if (r >= *nrows) return;
  const int kind = vi < NH ? 0 : (vi < NH + NKV ? 1 : 2), h = kind == 0 ? vi : (kind == 1 ? vi - NH : vi - NH - NKV);
  const int nd = D >> 5, half = D >> 1;
  const float* src = qkv + (size_t)r * qkv_dim + (kind == 0 ? h * D : NH * D + (kind == 2 ? NKV * D : 0) + h * D);
  float x[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) x[i] = i < nd ? __ldcg(src + lane + 32 * i) : 0.f;
  if (kind < 2) {
    if (qk_norm) {
      float ssq = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) ssq += x[i] * x[i];
#pragma unroll
      for (int off = 16; off; off >>= 1) ssq += __shfl_xor_sync(0xFFFFFFFFu, ssq, off);
      const float scl = rsqrtf(ssq / (float)D + eps);
      const float* gg = kind == 0 ? qn : kn;
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (i < nd) x[i] = x[i] * scl * __ldg(gg + lane + 32 * i);
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      if (i < nd / 2) {
        const float2 cs = __ldg(rope + (size_t)r * half + lane + 32 * i);
        const float a = x[i], b = x[i + nd / 2];
        x[i] = a * cs.x - b * cs.y;
        x[i + nd / 2] = b * cs.x + a * cs.y;
      }
    }
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    if (i < nd) {
      const int d = lane + 32 * i;
      if (kind == 0)
        q[(size_t)r * NH * D + h * D + d] = x[i];
      else
        (kind == 1 ? kc : vc)[((size_t)h * cap + r) * D + d] = (uint16_t)bf16_rn_bits(x[i]);
    }
  }
}

// Causal attention of the prompt rows over the bf16 cache: one warp per (row, query head),
// keys in blocks of 32 (lane j scores key j0 + j over all dims against the query in shared
// memory; running max and sum), P.V with lane owning dims lane + 32 i; the output row goes to
// the Wo operand (SW128 tiles, bf16).
__global__ void __launch_bounds__(256) pf_attn_kernel(const float* __restrict__ q, const int* nrows, int NH, int NKV,
                                                      int D, const uint16_t* __restrict__ kc,
                                                      const uint16_t* __restrict__ vc, int cap, int Rtc,
                                                      uint8_t* att_t) {
  __shared__ __align__(16) float qsh[8][128];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, w = blockIdx.x * 8 + warp;
  const int r = w / NH, h = w - r * NH;
  if (r >= *nrows) return;                  // whole warp
  const int g = h / (NH / NKV), nd = D >> 5;
  for (int d = lane; d < D; d += 32) qsh[warp][d] = __ldcg(q + (size_t)r * NH * D + h * D + d);
  __syncwarp();
  const float scale = rsqrtf((float)D);
  const uint16_t* kb = kc + (size_t)g * cap * D;
  const uint16_t* vb = vc + (size_t)g * cap * D;
  float m = -INFINITY, l = 0.f, acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int j0 = 0; j0 <= r; j0 += 32) {
    const int j = j0 + lane;
    float sc = -INFINITY;
    if (j <= r) {
      const uint4* kr = reinterpret_cast<const uint4*>(kb + (size_t)j * D);
      float a0 = 0.f, a1 = 0.f;
      for (int c = 0; c < D / 8; ++c) {
        const uint4 kk = __ldg(kr + c);
        const float* qq = qsh[warp] + 8 * c;
        a0 += qq[0] * bf16_lo_f32(kk.x) + qq[1] * bf16_hi_f32(kk.x) + qq[2] * bf16_lo_f32(kk.y) + qq[3] * bf16_hi_f32(kk.y);
        a1 += qq[4] * bf16_lo_f32(kk.z) + qq[5] * bf16_hi_f32(kk.z) + qq[6] * bf16_lo_f32(kk.w) + qq[7] * bf16_hi_f32(kk.w);
      }
      sc = (a0 + a1) * scale;
    }
    float mb = sc;
#pragma unroll
    for (int off = 16; off; off >>= 1) mb = fmaxf(mb, __shfl_xor_sync(0xFFFFFFFFu, mb, off));
    const float mn = fmaxf(m, mb);                       // finite: key j0 <= r is live
    const float corr = __expf(m - mn);
    const float pj = j <= r ? __expf(sc - mn) : 0.f;
    float ps = pj;
#pragma unroll
    for (int off = 16; off; off >>= 1) ps += __shfl_xor_sync(0xFFFFFFFFu, ps, off);
    l = l * corr + ps;
#pragma unroll
    for (int i = 0; i < 4; ++i) acc[i] *= corr;
    const int nk = min(32, r - j0 + 1);
    for (int jj = 0; jj < nk; ++jj) {
      const float pb = __shfl_sync(0xFFFFFFFFu, pj, jj);
      const uint16_t* vr = vb + (size_t)(j0 + jj) * D;
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (i < nd) acc[i] += pb * bf16_lo_f32((uint32_t)__ldg(vr + lane + 32 * i));
    }
    m = mn;
  }
  const float inv = 1.0f / l;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    if (i < nd) {
      const int f = h * D + lane + 32 * i;
      *reinterpret_cast<uint16_t*>(att_t + tc::sw128_offset(Rtc, r, f >> 6, (f & 63) >> 3) + (f & 7) * 2) =
          (uint16_t)bf16_rn_bits(acc[i] * inv);
    }
  }
}

struct mcd_outer {
  mcd_outer_config cfg;
  OuterTc tc;
  mcd_ctx* inner = nullptr;
  cudaStream_t stream = nullptr;
  FrameParams fp;
  OuterStep st;
  std::vector<void*> allocs;
  int P = 0;                    // codes per frame after c0 (the inner model's positions)
  int n_tok = 0;                // KV positions filled
  int frame = -1;               // frame whose c0 the last launch produced
  bool ready = false;           // that c0 has not yet started an inner frame
  bool weights_loaded = false;
  uint32_t stream_id = 0;
  int* c0_buf = nullptr;
  float* cond = nullptr;
  float* c0emb = nullptr;
  int* last_codes = nullptr;    // c0..c_P of the last frame a pipeline call decoded
  float* trace = nullptr;
  int trace_frames = 0;
};

template <class T>
static cudaError_t outer_alloc(mcd_outer* o, T** p, size_t bytes) {
  void* q = nullptr;
  cudaError_t e = cudaMalloc(&q, bytes < 256 ? 256 : bytes);
  if (e != cudaSuccess) return e;
  o->allocs.push_back(q);
  *p = static_cast<T*>(q);
  return cudaSuccess;
}

static mcd_status validate_outer(const mcd_outer_config& c, const FrameParams& ip) {
  if (c.n_layers < 1 || c.hidden != ip.H) return MCD_ERR_UNSUPPORTED;
  if (!(c.head_dim == 64 || c.head_dim == 128)) return MCD_ERR_UNSUPPORTED;
  if (c.n_q_heads < 1 || c.n_kv_heads < 1 || c.n_q_heads % c.n_kv_heads) return MCD_ERR_INVALID_ARG;
  if (c.n_q_heads / c.n_kv_heads > 8) return MCD_ERR_UNSUPPORTED;
  if (c.ffn < 128 || c.ffn % 128) return MCD_ERR_UNSUPPORTED;
  if ((long long)c.n_q_heads * c.head_dim + 2LL * c.n_kv_heads * c.head_dim > 8192) return MCD_ERR_UNSUPPORTED;
  if (c.c0_vocab < 16 || c.c0_vocab % 16 || c.c0_vocab > kMaxVocab) return MCD_ERR_UNSUPPORTED;
  if (c.text_vocab < 1) return MCD_ERR_INVALID_ARG;
  if (c.max_tokens < 1 || c.max_tokens > kMaxOuterTokens) return MCD_ERR_UNSUPPORTED;
  if (c.top_k < 1 || c.top_k > kMaxTopK || c.top_k > c.c0_vocab) return MCD_ERR_UNSUPPORTED;
  if (!(c.temperature > 0.f) || !(c.rms_eps > 0.f) || !(c.rope_base > 1.f)) return MCD_ERR_INVALID_ARG;
  if (c.weight_dtype != ip.wdtype) return MCD_ERR_INVALID_ARG;   // the frame sum reads the inner tables
  if (c.weight_dtype == MCD_WEIGHT_INT8) return MCD_ERR_UNSUPPORTED;
  if (ip.C0V != 0) return MCD_ERR_INVALID_ARG;                   // the inner model takes the c0 vector
  return MCD_OK;
}

static int prefill_rows(const mcd_outer* o) {
  return std::min(kMaxPrefillRows, kMaxQVec / (o->fp.NH / o->fp.NKV));
}

static mcd_status outer_launch(mcd_outer* o, const OuterStep& s) {
  FrameParams& p = o->fp;
  outer_begin_kernel<<<1, 256, 0, o->stream>>>(p.ctr, p.ctr_stride);
  MCD_CHECK(cudaGetLastError());
  void* args[] = {&p, const_cast<OuterStep*>(&s)};
  MCD_CHECK(cudaLaunchCooperativeKernel(outer_fn(p.wdtype, s.nr > kMaxRows), dim3(p.n_cta), dim3(kThreads), args,
                                        (size_t)kSmemBytes, o->stream));
  return MCD_OK;
}

// One CodeDecoder row for frame o->frame + 1 from the previous frame's codes (device).
static mcd_status outer_step_launch(mcd_outer* o, const int32_t* prev_codes, int32_t text_id, int32_t* c0_out2) {
  if (o->n_tok < 1) return MCD_ERR_STATE;
  if (o->n_tok >= o->st.cap) return MCD_ERR_STATE;   // the KV cache is full
  if (!prev_codes) return MCD_ERR_INVALID_ARG;
  if (text_id >= o->cfg.text_vocab) return MCD_ERR_INVALID_ARG;
  OuterStep s = o->st;
  s.pos0 = o->n_tok;
  s.nr = 1;
  s.head = 1;
  s.text_ids = nullptr;
  s.prev_codes = prev_codes;
  s.text_id = text_id < 0 ? -1 : text_id;
  s.c0_out2 = c0_out2;
  s.frame_id = (unsigned)(o->frame + 1);
  s.trace = (o->trace && o->frame + 1 < o->trace_frames)
                ? o->trace + (size_t)(o->frame + 1) * (o->fp.V + 2 * o->fp.H)
                : nullptr;
  mcd_status r = outer_launch(o, s);
  if (r != MCD_OK) return r;
  o->n_tok += 1;
  o->frame += 1;
  o->ready = true;
  return MCD_OK;
}

extern "C" {

mcd_status mcd_outer_create(const mcd_outer_config* cfg, mcd_ctx* inner, mcd_outer** out) {
  if (!out) return MCD_ERR_INVALID_ARG;
  *out = nullptr;
  if (!cfg || !inner) return MCD_ERR_INVALID_ARG;
  const FrameParams& ip = ctx_params(inner);
  mcd_status vs = validate_outer(*cfg, ip);
  if (vs != MCD_OK) return vs;
  mcd_outer* o = new mcd_outer();
  o->cfg = *cfg;
  o->inner = inner;
  o->stream = ctx_stream(inner);
  o->P = ip.P;
  auto fail = [&](mcd_status s) {
    mcd_outer_destroy(o);
    return s;
  };
  for (void* fn : {outer_fn(MCD_WEIGHT_BF16, false), outer_fn(MCD_WEIGHT_BF16, true), outer_fn(MCD_WEIGHT_F32, false),
                   outer_fn(MCD_WEIGHT_F32, true)})
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) != cudaSuccess)
      return fail(MCD_ERR_CUDA);
  const mcd_outer_config& k = *cfg;
  FrameParams& p = o->fp;
  memset(&p, 0, sizeof(p));
  p.L = k.n_layers;
  p.H = k.hidden;
  p.NH = k.n_q_heads;
  p.NKV = k.n_kv_heads;
  p.D = k.head_dim;
  p.F = k.ffn;
  p.P = ip.P;
  p.V = k.c0_vocab;
  p.C0V = k.c0_vocab;
  p.K = 0;
  p.top_k = k.top_k;
  p.qk_norm = k.qk_norm;
  p.wdtype = k.weight_dtype;
  p.eps = k.rms_eps;
  p.T = k.temperature;
  p.seed = k.seed;
  p.qkv_dim = p.NH * p.D + 2 * p.NKV * p.D;
  p.n_cta = ip.n_cta;
  p.wait_ns = ip.wait_ns;
  p.S = 1;
  if (!backbone_geom(p, p.V)) return fail(MCD_ERR_UNSUPPORTED);
  p.ctr_stride = ctr_count(p.L);
  const size_t es = k.weight_dtype == MCD_WEIGHT_BF16 ? 2 : 4;
  cudaError_t e;
  uint8_t *wq, *wo, *wg, *wd, *wh;
#define OUTER_ALLOC(ptr, bytes)                                              \
  do {                                                                       \
    if ((e = outer_alloc(o, &(ptr), (bytes))) != cudaSuccess) return fail(cuda_status(e)); \
  } while (0)
  OUTER_ALLOC(wq, (size_t)p.g[MAT_QKV].stride * p.L);
  OUTER_ALLOC(wo, (size_t)p.g[MAT_WO].stride * p.L);
  OUTER_ALLOC(wg, (size_t)p.g[MAT_GU].stride * p.L);
  OUTER_ALLOC(wd, (size_t)p.g[MAT_WD].stride * p.L);
  OUTER_ALLOC(wh, (size_t)p.g[MAT_HEAD].stride);
  p.w_qkv = wq;
  p.w_wo = wo;
  p.w_gu = wg;
  p.w_wd = wd;
  p.w_head = wh;
  float* f32 = nullptr;
  OUTER_ALLOC(f32, sizeof(float) * ((size_t)p.L * p.H * 2 + (size_t)p.L * p.D * 2 + p.H));
  p.attn_norm = f32;
  p.ffn_norm = p.attn_norm + (size_t)p.L * p.H;
  p.q_norm = p.ffn_norm + (size_t)p.L * p.H;
  p.k_norm = p.q_norm + (size_t)p.L * p.D;
  p.final_norm = p.k_norm + (size_t)p.L * p.D;
  OUTER_ALLOC(p.x, sizeof(float) * kMaxCols * p.H);
  OUTER_ALLOC(p.qkv, sizeof(float) * kMaxCols * p.qkv_dim);
  OUTER_ALLOC(p.mbuf, sizeof(float) * kMaxCols * p.F);
  OUTER_ALLOC(p.logits, sizeof(float) * p.V);
  OUTER_ALLOC(p.ctr, sizeof(unsigned) * p.ctr_stride);
  OUTER_ALLOC(p.err, sizeof(int));
  OuterStep& s = o->st;
  memset(&s, 0, sizeof(s));
  s.cap = k.max_tokens;
  const size_t kv = (size_t)p.L * p.NKV * s.cap * p.D * es;
  OUTER_ALLOC(s.kcache, kv);
  OUTER_ALLOC(s.vcache, kv);
  float2* rope = nullptr;
  OUTER_ALLOC(rope, sizeof(float2) * (size_t)s.cap * (p.D / 2));
  s.rope = rope;
  uint8_t *tt, *ct, *lt;
  OUTER_ALLOC(tt, (size_t)k.text_vocab * p.H * es);
  OUTER_ALLOC(ct, (size_t)k.c0_vocab * p.H * es);
  OUTER_ALLOC(lt, (size_t)ip.V * p.H * es);
  s.text_table = tt;
  s.text_vocab = k.text_vocab;
  s.c0_table = ct;
  s.c0_vocab = k.c0_vocab;
  s.code_tables = ip.embed;
  s.code_stride = ip.embed_stride;
  s.code_vocab = ip.V;
  s.P = ip.P;
  s.last_table = lt;
  const int n_blocks = (s.cap + kKeyBlock - 1) / kKeyBlock;
  OUTER_ALLOC(s.part, sizeof(float) * (size_t)n_blocks * kMaxPrefillRows * p.NH * kPartLd);
  OUTER_ALLOC(o->c0_buf, sizeof(int) * 4);
  OUTER_ALLOC(o->cond, sizeof(float) * p.H);
  OUTER_ALLOC(o->c0emb, sizeof(float) * p.H);
  OUTER_ALLOC(o->last_codes, sizeof(int) * (o->P + 1));
  OuterTc& t = o->tc;
  t.on = tc_block_supported(p) && s.cap >= 2;
  if (t.on) {
    const int Rtc = (s.cap + tc::kBM - 1) / tc::kBM * tc::kBM;
    t.Rtc = Rtc;
    t.off = tc_layer_offsets(p);
    OUTER_ALLOC(t.w, t.off.layer * p.L);
    OUTER_ALLOC(t.X, sizeof(float) * (size_t)Rtc * p.H);
    OUTER_ALLOC(t.ss, sizeof(float) * (size_t)Rtc);
    OUTER_ALLOC(t.qkv, sizeof(float) * (size_t)Rtc * p.qkv_dim);
    OUTER_ALLOC(t.q, sizeof(float) * (size_t)Rtc * p.NH * p.D);
    OUTER_ALLOC(t.part, sizeof(float) * (size_t)kTcSplit * Rtc * p.H);
    OUTER_ALLOC(t.xn_hi, (size_t)Rtc * p.H * 2);
    OUTER_ALLOC(t.xn_lo, (size_t)Rtc * p.H * 2);
    OUTER_ALLOC(t.att_t, (size_t)Rtc * p.NH * p.D * 2);
    OUTER_ALLOC(t.act_t, (size_t)Rtc * p.F * 2);
    OUTER_ALLOC(t.rows, sizeof(int));
    if (tc_block_set_smem() != cudaSuccess) return fail(MCD_ERR_CUDA);
  }
#undef OUTER_ALLOC
  s.c0_out = o->c0_buf;
  s.cond_out = o->cond;
  s.c0emb_out = o->c0emb;
  if (cudaMemsetAsync(p.err, 0, sizeof(int), o->stream) != cudaSuccess) return fail(MCD_ERR_CUDA);
  if (cudaMemsetAsync(s.kcache, 0, kv, o->stream) != cudaSuccess) return fail(MCD_ERR_CUDA);
  if (cudaMemsetAsync(s.vcache, 0, kv, o->stream) != cudaSuccess) return fail(MCD_ERR_CUDA);
  rope_kernel<<<64, 256, 0, o->stream>>>(rope, p.D, (double)k.rope_base, s.cap);
  if (cudaGetLastError() != cudaSuccess) return fail(MCD_ERR_CUDA);
  if (cudaStreamSynchronize(o->stream) != cudaSuccess) return fail(MCD_ERR_CUDA);
  *out = o;
  return MCD_OK;
}

void mcd_outer_destroy(mcd_outer* o) {
  if (!o) return;
  cudaStreamSynchronize(o->stream);
  for (void* q : o->allocs) cudaFree(q);
  delete o;
}

mcd_status mcd_outer_load_weights(mcd_outer* o, int32_t n, const char* const* names, const void* const* host_ptrs,
                                  const int64_t* nbytes) {
  if (!o || n <= 0 || !names || !host_ptrs || !nbytes) return MCD_ERR_INVALID_ARG;
  FrameParams& p = o->fp;
  const int64_t es = p.wdtype == MCD_WEIGHT_BF16 ? 2 : 4;
  std::map<std::string, std::pair<const void*, int64_t>> given;
  for (int i = 0; i < n; ++i) {
    if (!names[i] || !host_ptrs[i]) return MCD_ERR_INVALID_ARG;
    if (given.count(names[i])) return MCD_ERR_WEIGHTS;
    given[names[i]] = {host_ptrs[i], nbytes[i]};
  }
  const int64_t H = p.H, D = p.D, qd = (int64_t)p.NH * D, kd = (int64_t)p.NKV * D, F = p.F;
  auto have = [&](const std::string& name, int64_t count) {
    auto it = given.find(name);
    const bool ok = it != given.end() && it->second.second == count * es;
    if (!ok && getenv("MCD_DEBUG")) fprintf(stderr, "mcd: outer weight %s missing or wrong size\n", name.c_str());
    return ok;
  };
  // check every tensor before copying anything
  for (int l = 0; l < p.L; ++l) {
    const std::string pre = "layers." + std::to_string(l) + ".";
    if (!have(pre + "attn_norm", H) || !have(pre + "wq", qd * H) || !have(pre + "wk", kd * H) ||
        !have(pre + "wv", kd * H) || !have(pre + "wo", H * qd) || !have(pre + "ffn_norm", H) ||
        !have(pre + "wg", F * H) || !have(pre + "wu", F * H) || !have(pre + "wd", H * F))
      return MCD_ERR_WEIGHTS;
    if (p.qk_norm && (!have(pre + "q_norm", D) || !have(pre + "k_norm", D))) return MCD_ERR_WEIGHTS;
  }
  const std::string last = "code_embed." + std::to_string(o->P);
  if (!have("final_norm", H) || !have("c0_head", (int64_t)p.V * H) || !have("c0_embed", (int64_t)p.V * H) ||
      !have("text_embed", (int64_t)o->cfg.text_vocab * H) || !have(last, (int64_t)o->st.code_vocab * H))
    return MCD_ERR_WEIGHTS;
  // one layer's tensors (or the c0 head / final norm) at a time through a staging buffer
  const size_t layer_bytes = (size_t)(2 * H + 2 * D + qd * H + 2 * kd * H + H * qd + 3 * F * H) * es + 16 * 256;
  const size_t stage_bytes = std::max(layer_bytes, (size_t)(p.V * H + H) * es + 512);
  uint8_t* stage = nullptr;
  MCD_CHECK(cudaMalloc(&stage, stage_bytes));
  auto cleanup = [&](mcd_status s) {
    cudaStreamSynchronize(o->stream);
    cudaFree(stage);
    return s;
  };
  size_t off = 0;
  std::map<std::string, const uint8_t*> at;
  auto put = [&](const std::string& name) -> bool {
    auto& gv = given[name];
    if (cudaMemcpyAsync(stage + off, gv.first, (size_t)gv.second, cudaMemcpyHostToDevice, o->stream) != cudaSuccess)
      return false;
    at[name] = stage + off;
    off += ((size_t)gv.second + 255) / 256 * 256;
    return true;
  };
  for (int l = 0; l < p.L; ++l) {
    const std::string pre = "layers." + std::to_string(l) + ".";
    off = 0;
    at.clear();
    // the previous layer's tiling kernels read the staging buffer: wait for them
    if (cudaStreamSynchronize(o->stream) != cudaSuccess) return cleanup(MCD_ERR_CUDA);
    for (const char* t : {"wq", "wk", "wv", "wo", "wg", "wu", "wd", "attn_norm", "ffn_norm"})
      if (!put(pre + t)) return cleanup(MCD_ERR_CUDA);
    if (p.qk_norm && (!put(pre + "q_norm") || !put(pre + "k_norm"))) return cleanup(MCD_ERR_CUDA);
    LayerSrc ls{at[pre + "wq"], at[pre + "wk"], at[pre + "wv"], at[pre + "wo"], at[pre + "wg"], at[pre + "wu"],
                at[pre + "wd"], at[pre + "attn_norm"], at[pre + "ffn_norm"],
                p.qk_norm ? at[pre + "q_norm"] : nullptr, p.qk_norm ? at[pre + "k_norm"] : nullptr};
    load_layer(p, o->stream, ls, l);
    if (o->tc.on)
      tc_tile_layer(p, o->stream, ls.wq, ls.wk, ls.wv, ls.wo, ls.wg, ls.wu, ls.wd,
                    o->tc.w + (size_t)l * o->tc.off.layer);
  }
  if (cudaStreamSynchronize(o->stream) != cudaSuccess) return cleanup(MCD_ERR_CUDA);
  off = 0;
  at.clear();
  if (!put("c0_head") || !put("final_norm")) return cleanup(MCD_ERR_CUDA);
  RowSrc rh{};
  rh.seg[0] = at["c0_head"];
  rh.seg_rows[0] = p.V;
  rh.nseg = 1;
  rh.src_cols = (int)H;
  tile_kernel<<<1024, 256, 0, o->stream>>>(rh, p.g[MAT_HEAD], p.wdtype, const_cast<uint8_t*>(p.w_head), nullptr);
  to_f32_kernel<<<64, 256, 0, o->stream>>>(at["final_norm"], p.wdtype, H, const_cast<float*>(p.final_norm));
  // row-major tables go straight to their arrays
  auto table = [&](const std::string& name, const uint8_t* dst) {
    auto& gv = given[name];
    return cudaMemcpyAsync(const_cast<uint8_t*>(dst), gv.first, (size_t)gv.second, cudaMemcpyHostToDevice,
                           o->stream) == cudaSuccess;
  };
  if (!table("c0_embed", o->st.c0_table) || !table("text_embed", o->st.text_table) || !table(last, o->st.last_table))
    return cleanup(MCD_ERR_CUDA);
  if (cudaGetLastError() != cudaSuccess) return cleanup(MCD_ERR_CUDA);
  mcd_status s = cleanup(MCD_OK);
  if (cudaGetLastError() != cudaSuccess) return MCD_ERR_CUDA;
  o->weights_loaded = true;
  return s;
}

// Rows 0..n-1 of the prompt (positions 0..n-1) through every layer on the tensor cores,
// leaving their K / V in the cache.
static mcd_status outer_tc_prefill(mcd_outer* o, const int32_t* text_ids, int n) {
  const FrameParams& p = o->fp;
  const OuterTc& t = o->tc;
  const OuterStep& st = o->st;
  cudaStream_t s = o->stream;
  const int H = p.H, L = p.L, Rtc = t.Rtc, qd = p.NH * p.D, kvl = p.NKV * st.cap * p.D;
  const dim3 pblk(tc::kPThreads);
  pf_set_rows_kernel<<<1, 1, 0, s>>>(t.rows, n);
  pf_embed_kernel<<<n, 128, 0, s>>>(text_ids, t.rows, st.text_table, st.text_vocab, H, t.X, t.ss, p.err);
  tc_norm_operand_kernel<<<256, 256, 0, s>>>(t.X, p.attn_norm, t.ss, H, p.eps, t.rows, Rtc, t.xn_hi, t.xn_lo);
  for (int l = 0; l < L; ++l) {
    const uint8_t* wl = t.w + (size_t)l * t.off.layer;
    uint16_t* kc = reinterpret_cast<uint16_t*>(st.kcache) + (size_t)l * kvl;
    uint16_t* vc = reinterpret_cast<uint16_t*>(st.vcache) + (size_t)l * kvl;
    {
      const tc::GemmArgs g{wl + t.off.qkv, nullptr, t.xn_hi, t.xn_lo, p.qkv_dim, Rtc, H, t.rows, p.err, p.wait_ns};
      tc_qkv_kernel<<<tc_grid(tc_tiles(Rtc, kTcBN, p.qkv_dim, 1), p.n_cta), pblk, tc::PLayout<kTcBN, false, true>::kSmemBytes, s>>>(
          g, t.qkv, p.qkv_dim, t.rows);
    }
    const int vecs = p.NH + 2 * p.NKV;
    pf_rope_kv_kernel<<<(n * vecs + 7) / 8, 256, 0, s>>>(t.qkv, p.qkv_dim, t.rows, p.NH, p.NKV, p.D, p.qk_norm,
                                                         p.q_norm + (size_t)l * p.D, p.k_norm + (size_t)l * p.D, p.eps,
                                                         st.rope, kc, vc, st.cap, t.q);
    pf_attn_kernel<<<(n * p.NH + 7) / 8, 256, 0, s>>>(t.q, t.rows, p.NH, p.NKV, p.D, kc, vc, st.cap, Rtc, t.att_t);
    tc_launch_resid(wl + t.off.o, t.att_t, t.part, H, Rtc, qd, t.rows, p.err, p.wait_ns, p.n_cta, s);
    tc_resid_norm_kernel<<<n, 128, 0, s>>>(t.X, t.part, tc_splits(qd, tc_resid_split(Rtc)), Rtc, H, t.rows, t.ss, p.ffn_norm + (size_t)l * H,
                                           p.eps, t.xn_hi, nullptr);
    tc_launch_gu(wl + t.off.gu, t.xn_hi, t.act_t, Rtc, t.rows, p.F, H, p.err, p.wait_ns, p.n_cta, s);
    tc_launch_resid(wl + t.off.d, t.act_t, t.part, H, Rtc, p.F, t.rows, p.err, p.wait_ns, p.n_cta, s);
    tc_resid_norm_kernel<<<n, 128, 0, s>>>(t.X, t.part, tc_splits(p.F, tc_resid_split(Rtc)), Rtc, H, t.rows, t.ss,
                                           l + 1 < L ? p.attn_norm + (size_t)(l + 1) * H : nullptr, p.eps, t.xn_hi,
                                           t.xn_lo);
  }
  MCD_CHECK(cudaGetLastError());
  return MCD_OK;
}

mcd_status mcd_outer_prefill(mcd_outer* o, uint32_t stream_id, int32_t n_tokens, const int32_t* text_ids,
                             int32_t* c0_out) {
  if (!o || !text_ids || n_tokens < 1) return MCD_ERR_INVALID_ARG;
  if (!o->weights_loaded) return MCD_ERR_STATE;
  if (n_tokens > o->st.cap) return MCD_ERR_UNSUPPORTED;
  const int R = prefill_rows(o);
  o->stream_id = stream_id;
  o->st.stream_id = stream_id;
  // all but the last row on the tensor cores (when the shapes allow), the last through
  // outer_kernel (c0 head and sampling)
  int first = 0;
  if (o->tc.on && n_tokens >= 2) {
    mcd_status r = outer_tc_prefill(o, text_ids, n_tokens - 1);
    if (r != MCD_OK) return r;
    first = n_tokens - 1;
  }
  for (int s0 = first; s0 < n_tokens; s0 += R) {
    OuterStep s = o->st;
    s.pos0 = s0;
    s.nr = std::min(R, n_tokens - s0);
    s.head = s0 + s.nr == n_tokens ? 1 : 0;
    s.text_ids = text_ids + s0;
    s.prev_codes = nullptr;
    s.text_id = -1;
    s.c0_out2 = s.head ? c0_out : nullptr;
    s.frame_id = 0;
    s.trace = (o->trace && o->trace_frames > 0) ? o->trace : nullptr;
    mcd_status r = outer_launch(o, s);
    if (r != MCD_OK) return r;
  }
  o->n_tok = n_tokens;
  o->frame = 0;
  o->ready = true;
  return MCD_OK;
}

mcd_status mcd_outer_step(mcd_outer* o, const int32_t* prev_codes, int32_t text_id, int32_t* c0_out) {
  if (!o) return MCD_ERR_INVALID_ARG;
  if (!o->weights_loaded) return MCD_ERR_STATE;
  return outer_step_launch(o, prev_codes, text_id, c0_out);
}

mcd_status mcd_outer_frame_inputs(const mcd_outer* o, const float** cond, const float** c0_emb, const int32_t** c0,
                                  uint32_t* frame_idx) {
  if (!o) return MCD_ERR_INVALID_ARG;
  if (o->frame < 0) return MCD_ERR_STATE;
  if (cond) *cond = o->cond;
  if (c0_emb) *c0_emb = o->c0emb;
  if (c0) *c0 = o->c0_buf;
  if (frame_idx) *frame_idx = (uint32_t)o->frame;
  return MCD_OK;
}

mcd_status mcd_pipeline_frames(mcd_outer* o, int32_t n_frames, const int32_t* text_ids, int32_t* codes_out,
                               mcd_frame_stats* stats) {
  if (!o || n_frames < 0 || (!codes_out && n_frames > 0)) return MCD_ERR_INVALID_ARG;
  if (!o->weights_loaded || !ctx_weights_loaded(o->inner)) return MCD_ERR_STATE;
  if (o->frame < 0) return MCD_ERR_STATE;   // no prompt yet
  const int W = o->P + 1;
  for (int i = 0; i < n_frames; ++i) {
    int32_t* row = codes_out + (size_t)i * W;
    if (o->ready) {
      MCD_CHECK(cudaMemcpyAsync(row, o->c0_buf, sizeof(int32_t), cudaMemcpyDeviceToDevice, o->stream));
    } else {
      const int32_t* prev = i > 0 ? codes_out + (size_t)(i - 1) * W : o->last_codes;
      mcd_status r = outer_step_launch(o, prev, text_ids ? text_ids[i] : -1, row);
      if (r != MCD_OK) return r;
    }
    mcd_status r = mcd_decode_frame(o->inner, o->stream_id, (uint32_t)o->frame, o->cond, nullptr, o->c0emb, row + 1,
                                    stats ? stats + i : nullptr);
    if (r != MCD_OK) return r;
    o->ready = false;
  }
  if (n_frames > 0)
    MCD_CHECK(cudaMemcpyAsync(o->last_codes, codes_out + (size_t)(n_frames - 1) * W, sizeof(int32_t) * W,
                              cudaMemcpyDeviceToDevice, o->stream));
  return MCD_OK;
}

int64_t mcd_outer_trace_floats(const mcd_outer* o) { return o ? (int64_t)o->fp.V + 2LL * o->fp.H : 0; }

mcd_status mcd_outer_set_trace(mcd_outer* o, float* trace, int32_t n_frames) {
  if (!o || n_frames < 0 || (!trace && n_frames > 0)) return MCD_ERR_INVALID_ARG;
  o->trace = n_frames > 0 ? trace : nullptr;
  o->trace_frames = n_frames;
  return MCD_OK;
}

mcd_status mcd_outer_sync(mcd_outer* o) {
  if (!o) return MCD_ERR_INVALID_ARG;
  MCD_CHECK(cudaStreamSynchronize(o->stream));
  int err = 0;
  MCD_CHECK(cudaMemcpy(&err, o->fp.err, sizeof(int), cudaMemcpyDeviceToHost));
  return (mcd_status)err;
}

int64_t mcd_outer_step_weight_bytes(const mcd_outer* o) {
  if (!o) return 0;
  const FrameParams& p = o->fp;
  return (int64_t)p.L * (p.g[MAT_QKV].stride + p.g[MAT_WO].stride + p.g[MAT_GU].stride + p.g[MAT_WD].stride) +
         p.g[MAT_HEAD].stride;
}

}  // extern "C"
