// Persistent frame kernel: every model call of one frame of RVQ-position-aware
// speculative decoding (arXiv 2609.37007, Sec. 2.2 and Fig. 3) in a single cooperative
// launch with one CTA per SM.
//
// A launch decodes one frame for each of S streams (S = 1 for single-stream decoding); the
// streams advance in lock step, one call (round) at a time, and every call packs the rows of
// every stream whose frame is not finished into one operand (re-packed each round, since
// streams accept different numbers of drafts).
//
// Per call (a "round"): the rows [c_a, d_{a+1}, ..., d_{a+n}] (first call: [cond, c0]) go
// through the MultiCodeDecoder (5 pre-norm layers: RMSNorm -> QKV -> QK-norm -> RoPE ->
// causal GQA attention over the per-frame KV cache -> Wo + residual -> RMSNorm ->
// gate/up -> SwiGLU -> down + residual), the final RMSNorm gives h, LM head s reads row s
// (verify) and LM head s+j reads h_s + b_j (draft of position s+j).  Then the top-k /
// temperature distribution of every row, the acceptance step and the next drafts.
//
// The unit schedule, weight ring and unit GEMMs are in mcd_stage.cuh.
// The draft offsets enter as precomputed logit biases: LMH_P (h + b_j) = LMH_P h + LMH_P b_j,
// so every LM head multiplies the same operand (all rows' h).  Every wait is bounded.
#include "mcd_internal.cuh"
#include "mcd_sampler.cuh"
#include "mcd_stage.cuh"

namespace mcd {

// LM heads a pass reads, from the largest row position `top` of the pass.  Verify call:
// P_lo = a+1 up to top plus K (its draft heads), or up to top when the drafts come from
// noisy-target passes.  Noisy-target pass (one row at position top): head top only.
__device__ __forceinline__ void head_range(const FrameParams& p, int a, int top, int emu, int& p_lo, int& p_hi) {
  if (emu) {
    p_lo = p_hi = top;
    return;
  }
  p_lo = a + 1;
  p_hi = p.draft_mode == MCD_DRAFT_NOISY_TARGET ? top : min(p.P, top + p.K);
}

// LM heads one call streams: the union over the streams with rows in the call, as a bit
// mask over positions (bit P).
__device__ __forceinline__ unsigned call_heads_mask(const FrameParams& p) {
  unsigned mask = 0;
  for (int s = 0; s < p.S; ++s) {
    const DevState* st = p.st + s;
    if (__ldcg(&st->done)) continue;
    int lo, hi;
    head_range(p, __ldcg(&st->a), __ldcg(&st->top_pos), __ldcg(&st->emu), lo, hi);
    for (int P = lo; P <= hi; ++P) mask |= 1u << P;
  }
  return mask;
}

// ------------------------------------------------------------------------------------
// Producer: one thread streams this CTA's units into the ring.
// ------------------------------------------------------------------------------------
__device__ __forceinline__ void producer_loop(const FrameParams& p, Smem& sm, int call0) {
  const int cta = blockIdx.x, n_cta = p.n_cta;
  const uint64_t pol = policy_evict_first();
  uint32_t issued = 0;
  int rot = 0;
  volatile int* stop = sm.flags;
  bool halt = false;
  for (int call = call0; call < kMaxSlots && !halt; ++call) {
    int heads[16];
    for (int si = 0; si < n_stages(p) && !halt; ++si) {
      int n_heads = 0;
      if (stage_kind(si, p.L) == MAT_HEAD) {
        if (call != call0) {
          if (!wait_counter(p.ctr + call * p.ctr_stride + ctr_ready(p.L), 1u, p.err, p.wait_ns)) {
            halt = true;
            break;
          }
        }
        unsigned mask = call_heads_mask(p);
        if (!mask) {                       // every stream's frame is complete
          halt = true;
          break;
        }
        while (mask) {
          heads[n_heads++] = __ffs(mask) - 1;
          mask &= mask - 1;
        }
      }
      const int n = stage_units(p, si, n_heads);
      const uint32_t bytes = (uint32_t)p.g[stage_kind(si, p.L)].unit_bytes;
      const UnitRange ur = unit_range(si, p.L, n, cta, rot, n_cta);
      for (int u = ur.first; u < ur.end; u += ur.step) {
        if (!ring_issue(p, sm, issued, unit_src(p, si, u, heads), bytes, pol, stop)) {
          halt = true;
          break;
        }
      }
      rot = (rot + n) % n_cta;
    }
    if (p.single_call && !halt) {
      // a stepwise launch runs one verify call and the noisy-target passes that follow it
      if (!wait_counter(p.ctr + (call + 1) * p.ctr_stride + ctr_ready(p.L), 1u, p.err, p.wait_ns)) break;
      if (__ldcg(&p.st->emu) == 0 || __ldcg(&p.st->done)) break;
    }
  }
  ring_drain(p, sm, issued);
}


// Attention of query head h for the nr rows of stream s (packed rows base..base+nr-1; QK-norm,
// RoPE, causal softmax over the stream's per-frame cache plus the new rows); output
// o[base + n][D] in act.  Scratch spans act + bfrag
// (< 64 KB).  Phases, separated by barriers: (A) every input row (q, new k / v, cached
// k / v, RoPE rows, QK-norm gains) is loaded as independent 16-byte chunks, all in flight at
// once; (B) one warp per new q / k vector applies QK-norm and RoPE in registers (lane holds
// dims l + 32i, so each rotate-half pair (d, d + D/2) sits in one lane) and, for the KV
// writer, stores the new k / v rows to the cache; (C1) two threads per (row, key) score it
// over interleaved 16-byte chunks (rows padded to D + 8 floats: conflict-free reads); (C2)
// one warp per row takes the softmax; (C3) one thread per (row, dim pair) sums P.V.
__device__ __noinline__ void attention_stream(const FrameParams& p, int layer, int h, bool write_kv, int nr, int pos0, int base,
                                             int s) {
  Smem sm = smem_layout(mcd_dyn_smem);
  const int D = p.D, half = D >> 1, g = h / (p.NH / p.NKV);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int cs_shift = D == 128 ? 5 : 4;           // 16-byte chunks per row = D / 4
  const int cpr = 1 << cs_shift;
  const int KS = D + 8;                            // padded row stride (floats) of q and k rows
  constexpr int kAttnPos = 16;                     // sequence positions 0..15 (c15 is never fed)
  float* o = sm.act;                             // [kMaxCols][D]: every stream's packed rows
  float* qs = o + kMaxCols * 128;                  // [8][KS]
  float* ks = qs + kMaxRows * 136;                 // [kAttnPos][KS]
  float* vs = ks + kAttnPos * 136;                 // [kAttnPos][D]
  float2* cs = reinterpret_cast<float2*>(vs + kAttnPos * 128);  // [8][D/2] (cos, sin)
  float* gq = reinterpret_cast<float*>(cs + kMaxRows * 64);      // [D]
  float* gk = gq + 128;                                          // [D]
  const size_t cache_off = (size_t)s * p.kv_stride + ((size_t)layer * p.NKV + g) * p.kv_slots * D;
  const float* qkv = p.qkv;
  const int qoff = h * D, koff = p.NH * D + g * D, voff = p.NH * D + p.NKV * D + g * D;
  // ---- (A) loads ----------------------------------------------------------------------
  {
    const int n_new = nr << cs_shift, n_old = pos0 << cs_shift;
    const int e_q = n_new, e_k = 2 * n_new, e_v = 3 * n_new, e_kc = e_v + n_old, e_vc = e_kc + n_old;
    const int e_cs = e_vc + n_new, e_g = e_cs + (p.qk_norm ? 2 * cpr : 0);
    constexpr int kL = 10;
    float4 v[kL];
    float4* dst[kL];
#pragma unroll
    for (int u = 0; u < kL; ++u) {
      const int i = tid + u * kConsumerThreads;
      dst[u] = nullptr;
      if (i < e_g) {
        const float4* src;
        if (i < e_v) {
          const int seg = i < e_q ? 0 : (i < e_k ? 1 : 2);
          const int r = i - seg * n_new, n = r >> cs_shift, ch = r & (cpr - 1);
          src = reinterpret_cast<const float4*>(qkv + (size_t)(base + n) * p.qkv_dim +
                                                (seg == 0 ? qoff : seg == 1 ? koff : voff)) + ch;
          dst[u] = reinterpret_cast<float4*>(seg == 0 ? qs + n * KS : seg == 1 ? ks + (pos0 + n) * KS : vs + (pos0 + n) * D) + ch;
        } else if (i < e_vc) {
          const bool isk = i < e_kc;
          const int r = i - (isk ? e_v : e_kc), j = r >> cs_shift, ch = r & (cpr - 1);
          src = reinterpret_cast<const float4*>((isk ? p.kcache : p.vcache) + cache_off + (size_t)j * D) + ch;
          dst[u] = reinterpret_cast<float4*>(isk ? ks + j * KS : vs + j * D) + ch;
        } else if (i < e_cs) {
          const int r = i - e_vc, n = r >> cs_shift, ch = r & (cpr - 1);
          src = reinterpret_cast<const float4*>(p.rope + (size_t)(pos0 + n) * half) + ch;
          dst[u] = reinterpret_cast<float4*>(cs + n * 64) + ch;
        } else {
          const int r = i - e_cs, w = r >> cs_shift, ch = r & (cpr - 1);
          src = reinterpret_cast<const float4*>((w == 0 ? p.q_norm : p.k_norm) + (size_t)layer * D) + ch;
          dst[u] = reinterpret_cast<float4*>(w == 0 ? gq : gk) + ch;
        }
        v[u] = __ldcg(src);
      }
    }
#pragma unroll
    for (int u = 0; u < kL; ++u)
      if (dst[u]) *dst[u] = v[u];
  }
  consumer_sync();
  // ---- (B) QK-norm + RoPE of the new q / k rows; KV writer stores k / v ---------------
  const int nd = D >> 5;   // dims per lane: 4 (D = 128) or 2 (D = 64)
  for (int vi = warp; vi < 2 * nr; vi += kConsumerWarps) {
    const bool isq = vi < nr;
    const int n = isq ? vi : vi - nr;
    float* row = isq ? qs + n * KS : ks + (pos0 + n) * KS;
    float x[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) x[i] = i < nd ? row[lane + 32 * i] : 0.f;
    if (p.qk_norm) {
      float ss = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) ss += x[i] * x[i];
#pragma unroll
      for (int off = 16; off; off >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, off);
      const float sc = rsqrtf(ss / (float)D + p.eps);
      const float* gg = isq ? gq : gk;
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (i < nd) x[i] = x[i] * sc * gg[lane + 32 * i];
    }
    // rotate-half pairs: dims (lane + 32 i, lane + 32 i + D/2) for i < nd / 2
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      if (i < nd / 2) {
        const float2 r = cs[n * 64 + lane + 32 * i];
        const float a = x[i], b = x[i + nd / 2];
        x[i] = a * r.x - b * r.y;
        x[i + nd / 2] = b * r.x + a * r.y;
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (i < nd) row[lane + 32 * i] = x[i];
    if (write_kv) {
      float* kdst = p.kcache + cache_off + (size_t)(pos0 + n) * D;
      float* vdst = p.vcache + cache_off + (size_t)(pos0 + n) * D;
      if (!isq) {
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (i < nd) kdst[lane + 32 * i] = x[i];
      } else {
        const float* vrow = vs + (pos0 + n) * D;
#pragma unroll
        for (int i = 0; i < 4; ++i)
          if (i < nd) vdst[lane + 32 * i] = vrow[lane + 32 * i];
      }
    }
  }
  consumer_sync();
  // ---- (C1) scores: thread pair (n, j) splits the dot product over interleaved chunks ---
  float* sc = gk + 128;                            // [8][32] scores, then probabilities
  {
    const float scale = rsqrtf((float)D);
    for (int t = tid; t < (nr << 6); t += kConsumerThreads) {
      const int n = t >> 6, j = (t >> 1) & 31, hf = t & 1;
      const bool live = j <= pos0 + n;               // causal: keys 0..pos0+n
      float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
      if (live) {
        const float4* q4 = reinterpret_cast<const float4*>(qs + n * KS) + hf;
        const float4* k4 = reinterpret_cast<const float4*>(ks + j * KS) + hf;
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
      if (hf == 0) sc[n * 32 + j] = live ? acc * scale : -INFINITY;
    }
  }
  consumer_sync();
  // ---- (C2) softmax over the keys of row n: warp n ------------------------------------
  if (warp < nr) {
    const float s = sc[warp * 32 + lane];
    float m = s;
#pragma unroll
    for (int off = 16; off; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, off));
    const float e = lane <= pos0 + warp ? __expf(s - m) : 0.f;
    float sum = e;
#pragma unroll
    for (int off = 16; off; off >>= 1) sum += __shfl_xor_sync(0xFFFFFFFFu, sum, off);
    sc[warp * 32 + lane] = e / sum;
  }
  consumer_sync();
  // ---- (C3) o[n][d..d+1] = sum_j p_j v_j[d..d+1]: one thread per (row, dim pair) --------
  {
    const int lgh = D == 128 ? 6 : 5;              // dim pairs per row
    for (int t = tid; t < (nr << lgh); t += kConsumerThreads) {
      const int n = t >> lgh, d = 2 * (t & ((1 << lgh) - 1)), npos = pos0 + n + 1;
      const float* pr = sc + n * 32;
      float2 c0 = make_float2(0.f, 0.f), c1 = make_float2(0.f, 0.f);
      int j = 0;
      for (; j + 1 < npos; j += 2) {
        const float p0 = pr[j], p1 = pr[j + 1];
        const float2 v0 = *reinterpret_cast<const float2*>(vs + j * D + d);
        const float2 v1 = *reinterpret_cast<const float2*>(vs + (j + 1) * D + d);
        c0.x += p0 * v0.x;
        c0.y += p0 * v0.y;
        c1.x += p1 * v1.x;
        c1.y += p1 * v1.y;
      }
      if (j < npos) {
        const float p0 = pr[j];
        const float2 v0 = *reinterpret_cast<const float2*>(vs + j * D + d);
        c0.x += p0 * v0.x;
        c0.y += p0 * v0.y;
      }
      *reinterpret_cast<float2*>(o + (base + n) * D + d) = make_float2(c0.x + c1.x, c0.y + c1.y);
    }
  }
  consumer_sync();
}


// Attention of query head h for the nr rows of stream s (packed rows base..base+nr-1), the
// single-stream form; same outputs and cache writes as attention_stream (o[base + n][D] in
// act).  (A) all threads stage the stream's cached K / V rows, the new rows' raw q / k / v,
// their RoPE rows and the QK-norm gains in shared memory (independent 16-byte loads, all in
// flight together); (B) one warp per new q / k vector applies QK-norm and RoPE in registers
// (lane l holds dims l + 32 i, so each rotate-half pair sits in one lane) and the KV writer
// stores the new keys and values; (C) the warp of query row n scores its keys with two lanes
// per key (interleaved 16-byte chunks, one shuffle), takes the softmax across its lanes and
// sums P.V with four dims per lane.  Three barriers in all; keys: positions 0..15 (c15 is
// never fed).
constexpr int kAttnKeys = 16;
__device__ __noinline__ void attention_rows(const FrameParams& p, int layer, int h, bool write_kv, int nr, int pos0, int base,
                                           int s) {
  Smem sm = smem_layout(mcd_dyn_smem);
  const int D = p.D, half = D >> 1, g = h / (p.NH / p.NKV);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int cs_shift = D == 128 ? 5 : 4, cpr = 1 << cs_shift;   // 16-byte chunks per row
  constexpr int KS = 136;                                       // padded q / k row stride
  float* o = sm.act;                                          // [kMaxCols][D]
  float* ks = o + kMaxCols * 128;                               // [kAttnKeys][KS]
  float* vs = ks + kAttnKeys * KS;                              // [kAttnKeys][128]
  float* qs = vs + kAttnKeys * 128;                             // [kMaxRows][KS]
  float2* cs = reinterpret_cast<float2*>(qs + kMaxRows * KS);   // [kMaxRows][D/2]
  float* gq = reinterpret_cast<float*>(cs + kMaxRows * 64);     // [D]
  float* gk = gq + 128;                                         // [D]
  const size_t cache_off = (size_t)s * p.kv_stride + ((size_t)layer * p.NKV + g) * p.kv_slots * D;
  const float* qkv = p.qkv;
  const int qoff = h * D, koff = p.NH * D + g * D, voff = p.NH * D + p.NKV * D + g * D;
  if (pos0 + nr > kAttnKeys) {                // positions beyond c14's row are never fed
    if (tid == 0) atomicCAS(p.err, 0, (int)MCD_ERR_STATE);
    nr = max(0, kAttnKeys - pos0);
  }
  // ---- (A) staging: rows [cached K | cached V | q | k | v | RoPE | gains], 16-byte chunks --
  {
    const int n_rows = 2 * pos0 + 4 * nr + (p.qk_norm ? 2 : 0);
    for (int i = tid; i < (n_rows << cs_shift); i += kConsumerThreads) {
      int r = i >> cs_shift;
      const int ch = i & (cpr - 1);
      const float* src;
      float* dst;
      if (r < 2 * pos0) {
        const bool isv = r >= pos0;
        const int j = isv ? r - pos0 : r;
        src = (isv ? p.vcache : p.kcache) + cache_off + (size_t)j * D;
        dst = isv ? vs + j * 128 : ks + j * KS;
      } else if ((r -= 2 * pos0) < 3 * nr) {
        const int seg = r >= 2 * nr ? 2 : r >= nr ? 1 : 0, m = r - seg * nr;
        src = qkv + (size_t)(base + m) * p.qkv_dim + (seg == 0 ? qoff : seg == 1 ? koff : voff);
        dst = seg == 0 ? qs + m * KS : seg == 1 ? ks + (pos0 + m) * KS : vs + (pos0 + m) * 128;
      } else if ((r -= 3 * nr) < nr) {
        src = reinterpret_cast<const float*>(p.rope + (size_t)(pos0 + r) * half);
        dst = reinterpret_cast<float*>(cs + r * 64);
      } else {
        r -= nr;
        src = (r == 0 ? p.q_norm : p.k_norm) + (size_t)layer * D;
        dst = r == 0 ? gq : gk;
      }
      cpa16(dst + 4 * ch, src + 4 * ch);
    }
    cpa_wait_all();
  }
  consumer_sync();
  // ---- (B) QK-norm + RoPE of the new q / k rows; the KV writer stores k / v -------------
  const int nd = D >> 5;   // dims per lane: 4 (D = 128) or 2 (D = 64)
  for (int vi = warp; vi < 2 * nr; vi += kConsumerWarps) {
    const bool isq = vi < nr;
    const int n = isq ? vi : vi - nr;
    float* row = isq ? qs + n * KS : ks + (pos0 + n) * KS;
    float x[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) x[i] = i < nd ? row[lane + 32 * i] : 0.f;
    if (p.qk_norm) {
      float ss = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) ss += x[i] * x[i];
#pragma unroll
      for (int off = 16; off; off >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, off);
      const float sc = rsqrtf(ss / (float)D + p.eps);
      const float* gg = isq ? gq : gk;
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (i < nd) x[i] = x[i] * sc * gg[lane + 32 * i];
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      if (i < nd / 2) {
        const float2 r = cs[n * 64 + lane + 32 * i];
        const float a = x[i], b = x[i + nd / 2];
        x[i] = a * r.x - b * r.y;
        x[i + nd / 2] = b * r.x + a * r.y;
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (i < nd) row[lane + 32 * i] = x[i];
    if (write_kv && !isq) {
      float* kdst = p.kcache + cache_off + (size_t)(pos0 + n) * D;
      float* vdst = p.vcache + cache_off + (size_t)(pos0 + n) * D;
      const float* vrow = vs + (pos0 + n) * 128;
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (i < nd) {
          kdst[lane + 32 * i] = x[i];
          vdst[lane + 32 * i] = vrow[lane + 32 * i];
        }
    }
  }
  consumer_sync();
  // ---- (C) warp n: scores (lanes 2j, 2j+1 for key j), softmax, P.V -----------------------
  if (warp < nr) {
    const int n = warp, npos = pos0 + n + 1;
    const int j = lane >> 1, hf = lane & 1;
    const bool live = j < npos;                      // causal: keys 0..pos0+n
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
    if (live) {
      const float4* q4 = reinterpret_cast<const float4*>(qs + n * KS) + hf;
      const float4* k4 = reinterpret_cast<const float4*>(ks + j * KS) + hf;
#pragma unroll 4
      for (int ch = 0; ch < (cpr >> 1); ++ch) {
        const float4 q = q4[2 * ch], k = k4[2 * ch];
        a0 += q.x * k.x;
        a1 += q.y * k.y;
        a2 += q.z * k.z;
        a3 += q.w * k.w;
      }
    }
    float sc = (a0 + a1) + (a2 + a3);
    sc += __shfl_xor_sync(0xFFFFFFFFu, sc, 1);
    sc = live ? sc * rsqrtf((float)D) : -INFINITY;
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
#pragma unroll 4
    for (int jj = 0; jj < npos; ++jj) {
      const float w = __shfl_sync(0xFFFFFFFFu, pj, 2 * jj);
      if (d0 < D) {
        const float4 v = *reinterpret_cast<const float4*>(vs + jj * 128 + d0);
        acc.x += w * v.x;
        acc.y += w * v.y;
        acc.z += w * v.z;
        acc.w += w * v.w;
      }
    }
    if (d0 < D) *reinterpret_cast<float4*>(o + (base + n) * D + d0) = acc;
  }
  consumer_sync();
}

// Attention of query head h for every stream with rows in the call (outputs at the
// streams' packed rows).
__device__ void attention_head(Cons& c, int layer, int h, bool write_kv) {
  const CallInfo* ci = c.sm.ci;
  for (int i = 0; i < ci->n_act; ++i) {
    const int s = ci->act[i];
    attention_rows(c.p, layer, h, write_kv, ci->st[s].n_rows, ci->st[s].pos0, ci->base[s], s);
  }
}

// Attention of query head h for rows lo..hi-1 of the current pass of a tree call (one
// stream; pass row n is tree row row0 + n).  Tree row m >= 1 is node m - 1 at position
// pos0 + depth; row 0 feeds the last emitted code at pos0.  A query row sees the committed
// positions 0..pos0-1, row 0, its ancestors and itself (the sparse tree mask of Fig. 2).
// Keys, compacted: positions 0..pos0-1 (cache slots), then the tree rows visible to at
// least one query of the group, in tree order.  Rows of earlier passes come from the cache
// (row 0 at slot pos0, node rows at kMaxPos + m), already normalised and rotated; rows of
// this pass come from the QKV output and are normalised and rotated here at their own
// position.  The task of a KV head's first query head stores K / V of rows lo..hi-1.
// Outputs go to p.attn (pass rows).  Scratch (act + bfrag, 62.6 KB): k [48][D + 8],
// v [48][D], q [8][D + 8], RoPE rows by depth [8][D/2], QK-norm gains, scores [8][48],
// the key rows and the queries' ancestor masks.
__device__ __noinline__ void attention_tree_task(const FrameParams& p, int layer, int h, int lo, int hi, int pos0) {
  Smem sm = smem_layout(mcd_dyn_smem);
  const CallInfo* ci = sm.ci;
  const int D = p.D, half = D >> 1, group = p.NH / p.NKV, g = h / group, row0 = ci->row0;
  const bool write_kv = (h % group) == 0;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int cs_shift = D == 128 ? 5 : 4, cpr = 1 << cs_shift;   // 16-byte chunks per row
  const int KS = D + 8;
  constexpr int kKeys = kTreeKeys, kDepths = kMaxDraft + 1;
  float* ks = sm.act;
  float* vs = ks + kKeys * 136;
  float* qs = vs + kKeys * 128;
  float2* cs = reinterpret_cast<float2*>(qs + 8 * 136);
  float* gq = reinterpret_cast<float*>(cs + kDepths * 64);
  float* gk = gq + 128;
  float* sc = gk + 128;
  unsigned long long* qanc = reinterpret_cast<unsigned long long*>(sc + 8 * kKeys);   // [8]
  int* krow = reinterpret_cast<int*>(qanc + 8);                  // [kKeys - pos0] tree row of key pos0 + i
  __shared__ int s_nk, s_jc;
  const size_t cache_off = ((size_t)layer * p.NKV + g) * p.kv_slots * D;
  const float* qkv = p.qkv;
  const int qoff = h * D, koff = p.NH * D + g * D, voff = p.NH * D + p.NKV * D + g * D;
  const int nq = hi - lo, dm = min(p.tree_maxd, kMaxPos - 1 - pos0);   // RoPE rows pos0 .. pos0 + dm
  // ---- key list: row 0 and the union of the queries' ancestor-or-self sets -----------------
  if (tid == 0) {
    unsigned long long U = 0ull;
    for (int n = lo; n < hi; ++n) {
      const int m = row0 + n;
      const unsigned long long am = m > 0 ? p.tree_anc[m - 1] : 0ull;
      qanc[n - lo] = am;
      U |= am;
    }
    int nk = pos0, jc = -1;
    krow[0] = 0;
    ++nk;
    if (row0 == 0) jc = pos0;
    while (U) {
      const int m = __ffsll((long long)U);                       // node m - 1 -> tree row m
      U &= U - 1ull;
      if (nk >= kKeys) {                                           // groups are sized to fit
        atomicCAS(p.err, 0, (int)MCD_ERR_STATE);
        break;
      }
      if (jc < 0 && m >= row0) jc = nk;
      krow[nk - pos0] = m;
      ++nk;
    }
    s_nk = nk;
    s_jc = jc < 0 ? nk : jc;                                       // keys jc.. are rows of this pass
  }
  consumer_sync();
  const int nk = s_nk, jc = s_jc;
  auto key_slot = [&](int j) {                                    // cache slot of an earlier key
    if (j < pos0) return j;
    const int m = krow[j - pos0];
    return m == 0 ? pos0 : kMaxPos + m;
  };
  auto row_depth = [&](int m) { return m == 0 ? 0 : (int)p.tree_depth[m - 1]; };
  // ---- (A) loads, 16-byte chunks, batches of 8 per thread in flight --------------------------
  {
    const int e_q = nq << cs_shift, e_k = e_q + (nk << cs_shift), e_v = e_k + (nk << cs_shift);
    const int e_cs = e_v + ((dm + 1) << cs_shift), e_g = e_cs + (p.qk_norm ? 2 * cpr : 0);
    for (int base = 0; base < e_g; base += 8 * kConsumerThreads) {
      float4 v[8];
      float4* dst[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int i = base + tid + u * kConsumerThreads;
        dst[u] = nullptr;
        if (i >= e_g) continue;
        const float4* src;
        const int ch = i & (cpr - 1);
        if (i < e_q) {
          const int n = lo + (i >> cs_shift);
          src = reinterpret_cast<const float4*>(qkv + (size_t)n * p.qkv_dim + qoff);
          dst[u] = reinterpret_cast<float4*>(qs + (n - lo) * KS) + ch;
        } else if (i < e_v) {
          const bool isv = i >= e_k;
          const int j = (i - (isv ? e_k : e_q)) >> cs_shift;
          if (j >= jc)
            src = reinterpret_cast<const float4*>(qkv + (size_t)(krow[j - pos0] - row0) * p.qkv_dim +
                                                  (isv ? voff : koff));
          else
            src = reinterpret_cast<const float4*>((isv ? p.vcache : p.kcache) + cache_off +
                                                  (size_t)key_slot(j) * D);
          dst[u] = reinterpret_cast<float4*>(isv ? vs + j * D : ks + j * KS) + ch;
        } else if (i < e_cs) {
          const int d = (i - e_v) >> cs_shift;
          src = reinterpret_cast<const float4*>(p.rope + (size_t)(pos0 + d) * half);
          dst[u] = reinterpret_cast<float4*>(cs + d * 64) + ch;
        } else {
          const int w = (i - e_cs) >> cs_shift;
          src = reinterpret_cast<const float4*>((w == 0 ? p.q_norm : p.k_norm) + (size_t)layer * D);
          dst[u] = reinterpret_cast<float4*>(w == 0 ? gq : gk) + ch;
        }
        v[u] = __ldcg(src + ch);
      }
#pragma unroll
      for (int u = 0; u < 8; ++u)
        if (dst[u]) *dst[u] = v[u];
    }
  }
  consumer_sync();
  // ---- (B) QK-norm + RoPE of the queries and this pass's keys; K / V of rows lo..hi-1 stored ---
  const int nd = D >> 5;
  for (int vi = warp; vi < nq + nk - jc; vi += kConsumerWarps) {
    const bool isq = vi < nq;
    const int j = jc + vi - nq;                                   // key index (keys only)
    const int m = isq ? row0 + lo + vi : krow[j - pos0];          // tree row
    float* row = isq ? qs + vi * KS : ks + j * KS;
    const int depth = row_depth(m);
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
        const float2 r = cs[depth * 64 + lane + 32 * i];
        const float a0 = x[i], b0 = x[i + nd / 2];
        x[i] = a0 * r.x - b0 * r.y;
        x[i + nd / 2] = b0 * r.x + a0 * r.y;
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (i < nd) row[lane + 32 * i] = x[i];
    const int n = m - row0;                                       // pass row of a key
    if (!isq && write_kv && n >= lo && n < hi) {
      const int slot = m == 0 ? pos0 : kMaxPos + m;
      float* kd = p.kcache + cache_off + (size_t)slot * D;
      float* vd = p.vcache + cache_off + (size_t)slot * D;
      const float* vrow = vs + j * D;
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (i < nd) {
          kd[lane + 32 * i] = x[i];
          vd[lane + 32 * i] = vrow[lane + 32 * i];
        }
    }
  }
  consumer_sync();
  // ---- (C1) scores: two threads per (query, key) over interleaved chunks ----------------------
  {
    const float scale = rsqrtf((float)D);
    for (int t = tid; t < nq * kKeys * 2; t += kConsumerThreads) {
      const int qi = t / (2 * kKeys), j = (t >> 1) % kKeys, hf = t & 1;
      bool live = j < nk;
      if (live && j > pos0) live = (qanc[qi] >> (krow[j - pos0] - 1)) & 1ull;   // j == pos0: row 0
      float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
      if (live) {
        const float4* q4 = reinterpret_cast<const float4*>(qs + qi * KS) + hf;
        const float4* k4 = reinterpret_cast<const float4*>(ks + j * KS) + hf;
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
      if (hf == 0) sc[qi * kKeys + j] = live ? acc * scale : -INFINITY;
    }
  }
  consumer_sync();
  // ---- (C2) softmax: one warp per query, keys lane and lane + 32 ---------------------------------
  for (int qi = warp; qi < nq; qi += kConsumerWarps) {
    const float s0 = sc[qi * kKeys + lane];
    const float s1 = lane + 32 < kKeys ? sc[qi * kKeys + lane + 32] : -INFINITY;
    float m = fmaxf(s0, s1);
#pragma unroll
    for (int off = 16; off; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, off));
    const float e0 = s0 == -INFINITY ? 0.f : __expf(s0 - m), e1 = s1 == -INFINITY ? 0.f : __expf(s1 - m);
    float l = e0 + e1;
#pragma unroll
    for (int off = 16; off; off >>= 1) l += __shfl_xor_sync(0xFFFFFFFFu, l, off);
    sc[qi * kKeys + lane] = e0 / l;
    if (lane + 32 < kKeys) sc[qi * kKeys + lane + 32] = e1 / l;
  }
  consumer_sync();
  // ---- (C3) o = sum_j p_j v_j over the keys (masked keys have p_j = 0) ----------------------
  for (int t = tid; t < nq * half; t += kConsumerThreads) {
    const int qi = t / half, d = 2 * (t - qi * half), n = lo + qi;
    const float* pr = sc + qi * kKeys;
    float2 acc = make_float2(0.f, 0.f);
    for (int j = 0; j < nk; ++j) {
      const float w = pr[j];
      const float2 v = *reinterpret_cast<const float2*>(vs + j * D + d);
      acc.x += w * v.x;
      acc.y += w * v.y;
    }
    *reinterpret_cast<float2*>(p.attn + (size_t)n * p.NH * D + h * D + d) = acc;
  }
  consumer_sync();
}

// ------------------------------------------------------------------------------------
// One call
// ------------------------------------------------------------------------------------
template <int WT, bool WIDE>
__device__ __forceinline__ void run_call(Cons& c, int call) {
  const FrameParams& p = c.p;
  Smem& sm = c.sm;
  const CallInfo* ci = sm.ci;
  const int L = p.L, H = p.H, D = p.D, F = p.F;
  unsigned* ctr = p.ctr + (size_t)call * p.ctr_stride;
  const int n_rows = ci->M;                 // packed rows of every stream in the call
  const unsigned N = (unsigned)p.n_cta;
  const float* x = p.x;
  auto from_x = [&](int n, int k, auto w) { return ld_global_v<decltype(w)::value>(x + (size_t)n * H + k); };

  auto no_key = [](int) { return 0; };
  auto no_prep = [](int, int, int) {};
  for (int l = 0; l < L; ++l) {
    // ---- S1: RMSNorm -> QKV  (q, k, v = W (x . g) / rms) -------------------------------
    g2s_vec(sm.vec, p.attn_norm + (size_t)l * H, H);      // independent of the wait below
    const StagePlan sp_qkv = plan_stage<WT, WIDE>(c, 4 * l + 0, p.g[MAT_QKV].n_units, n_rows, no_key);
    if (l == 0) {
      // layer-0 rows straight from their sources (cond / c0 vector / embedding rows); CTA 0
      // also seeds the residual stream x
      consumer_sync();                     // the gain is in shared memory
      prep_operand<WT, WIDE>(
          c, n_rows, H, 0, H, sm.vec, true,
          [&](int n, int k, auto w) {
            constexpr int W = decltype(w)::value;
            const uint8_t* src = ci->r_src[n];
            return ci->r_f32[n] ? ldg_f32_v<W>(src, k) : ldg_bf16_v<W>(src, k);
          },
          blockIdx.x == 0 ? p.x : nullptr);
    } else {
      if (!cons_wait(c, ctr + ctr_stage(l - 1, 3), N)) return;
      prep_operand<WT, WIDE>(c, n_rows, H, 0, H, sm.vec, true, from_x);
    }
    {
      const MatGeom& g = p.g[MAT_QKV];
      run_stage<WT, WIDE>(c, call, sp_qkv, H, no_key, no_prep,
                    [&](int u, int mi, int rr, int n, float v, float) {
                      const int row = (u % g.n_mb) * g.Mu * 16 + mi * 16 + rr;
                      p.qkv[(size_t)n * p.qkv_dim + row] = v * sm.inv_rms[n] * wscale<WT>(p.s_qkv, (size_t)l * p.qkv_dim + row);
                    });
      if (c.abort_) return;
    }
    cons_signal(c, ctr + ctr_stage(l, 0), call, 10 + 4 * (4 * l + 0));

    // ---- S2: attention (per query head) -> Wo + residual --------------------------------
    // Unit u of Wo covers m-block u % n_mb of query head h = u / n_mb (its k-chunk); its B
    // operand is head h's attention output.  Single stream: the CTAs holding head h's Wo
    // units compute that attention themselves.  Several streams: first one task per
    // (stream, query head) spread over the CTAs writes the outputs to global memory, then
    // Wo reads them.
    auto wo_key = [&](int u) { return u / p.g[MAT_WO].n_mb; };
    const StagePlan sp_wo = plan_stage<WT, WIDE>(c, 4 * l + 1, p.g[MAT_WO].n_units, n_rows, wo_key);
    if (!WIDE && threadIdx.x == 0) sm.flags[3] = -1;     // ordered by the wait's barrier
    if (!cons_wait(c, ctr + ctr_stage(l, 0), N)) return;
    if (WIDE) {
      if (p.draft_mode == MCD_DRAFT_TREE && ci->st[0].pos0 > 0) {
        // tree call (one stream): one task per (query head, row group of the pass)
        for (int t = blockIdx.x; t < p.NH * ci->n_tg; t += p.n_cta) {
          const int gi = t / p.NH;
          attention_tree_task(p, l, t - gi * p.NH, ci->tg[gi], ci->tg[gi + 1], ci->st[0].pos0);
        }
      } else {
        const int group = p.NH / p.NKV, n_tasks = ci->n_act * p.NH;
        for (int t = blockIdx.x; t < n_tasks; t += p.n_cta) {
          const int i = t / p.NH, h = t - i * p.NH, s = ci->act[i];
          const int nr = ci->st[s].n_rows, base = ci->base[s];
          attention_stream(p, l, h, (h % group) == 0, nr, ci->st[s].pos0, base, s);
          for (int q = threadIdx.x; q < nr * (D >> 2); q += kConsumerThreads) {
            const int n = q / (D >> 2), d4 = q - n * (D >> 2);
            reinterpret_cast<float4*>(p.attn + (size_t)(base + n) * p.NH * D + h * D)[d4] =
                reinterpret_cast<const float4*>(sm.act + (base + n) * D)[d4];
          }
          consumer_sync();
        }
      }
      cons_signal(c, ctr + ctr_att(L, l), call, kTimelineSlots);
      if (!cons_wait(c, ctr + ctr_att(L, l), N)) return;
      const MatGeom& g = p.g[MAT_WO];
      if (threadIdx.x == 0) sm.flags[3] = -1;
      consumer_sync();
      run_stage<WT, WIDE, true>(
          c, call, sp_wo, D, wo_key,
          [&](int u, int, int) {
            const int h = u / g.n_mb;
            if (sm.flags[3] != h) {
              const float* src = p.attn + h * D;
              prep_operand<WT, WIDE>(c, n_rows, D, 0, D, nullptr, false,
                                     [&](int n, int k, auto w) { return ld_global_v<decltype(w)::value>(src + (size_t)n * p.NH * D + k); });
              if (threadIdx.x == 0) sm.flags[3] = h;
            }
          },
          [&](int u, int mi, int rr0, int n, float4 v) {
            const int row = (u % g.n_mb) * g.Mu * 16 + mi * 16 + rr0;
            const size_t si = (size_t)l * H + row;
            red_add_f32x4(p.x + (size_t)n * H + row,
                          make_float4(v.x * wscale<WT>(p.s_wo, si), v.y * wscale<WT>(p.s_wo, si + 1),
                                      v.z * wscale<WT>(p.s_wo, si + 2), v.w * wscale<WT>(p.s_wo, si + 3)));
          });
      if (c.abort_) return;
    } else {
      const MatGeom& g = p.g[MAT_WO];
      const int group = p.NH / p.NKV;
      run_stage<WT, WIDE, true>(
          c, call, sp_wo, D, wo_key,
          [&](int u, int cnt, int step) {
            const int h = u / g.n_mb;
            bool writer = false;      // the CTA holding m-block 0 of a group's first head writes K / V
            for (int r = 0; r < cnt; ++r) writer |= (h % group) == 0 && (u + r * step) % g.n_mb == 0;
            if (sm.flags[3] != h || writer) {
              attention_head(c, l, h, writer);
              c.op = reinterpret_cast<uint8_t*>(sm.act) + kWoOperandOff;
              prep_operand<WT, WIDE>(c, n_rows, D, 0, D, nullptr, false,
                               [&](int n, int k, auto w) { return ld_shared_v<decltype(w)::value>(sm.act + n * D + k); });
              if (threadIdx.x == 0) sm.flags[3] = h;
            }
          },
          [&](int u, int mi, int rr0, int n, float4 v) {
            const int row = (u % g.n_mb) * g.Mu * 16 + mi * 16 + rr0;
            const size_t si = (size_t)l * H + row;
            red_add_f32x4(p.x + (size_t)n * H + row,
                          make_float4(v.x * wscale<WT>(p.s_wo, si), v.y * wscale<WT>(p.s_wo, si + 1),
                                      v.z * wscale<WT>(p.s_wo, si + 2), v.w * wscale<WT>(p.s_wo, si + 3)));
          });
      if (c.abort_) return;
    }
    c.op = reinterpret_cast<uint8_t*>(sm.act);
    cons_signal(c, ctr + ctr_stage(l, 1), call, 10 + 4 * (4 * l + 1));

    // ---- S3: RMSNorm -> gate/up -> SwiGLU --------------------------------------------------
    g2s_vec(sm.vec, p.ffn_norm + (size_t)l * H, H);
    const StagePlan sp_gu = plan_stage<WT, WIDE>(c, 4 * l + 2, p.g[MAT_GU].n_units, n_rows, no_key, true);
    if (!cons_wait(c, ctr + ctr_stage(l, 1), N)) return;
    prep_operand<WT, WIDE>(c, n_rows, H, 0, H, sm.vec, true, from_x);
    {
      const MatGeom& g = p.g[MAT_GU];
      // tile rows 0..7 are gate rows j0..j0+7, rows 8..15 the matching up rows
      run_stage<WT, WIDE>(
          c, call, sp_gu, H, no_key, no_prep,
          [&](int u, int mi, int rr, int n, float gate, float up) {
            const float s = sm.inv_rms[n];
            const int t16 = ((u % g.n_mb) * g.Mu + mi) * 16 + rr;      // tiled row of the gate
            const float gt = gate * s * wscale<WT>(p.s_gu, (size_t)l * 2 * F + t16);
            const float ut = up * s * wscale<WT>(p.s_gu, (size_t)l * 2 * F + t16 + 8);
            const int j = ((u % g.n_mb) * g.Mu + mi) * 8 + rr;
            p.mbuf[(size_t)n * F + j] = gt / (1.0f + __expf(-gt)) * ut;
          });
      if (c.abort_) return;
    }
    cons_signal(c, ctr + ctr_stage(l, 2), call, 10 + 4 * (4 * l + 2));

    // ---- S4: down + residual (k-chunks of F) ---------------------------------------------
    auto wd_key = [&](int u) { return u / p.g[MAT_WD].n_mb; };
    const StagePlan sp_wd = plan_stage<WT, WIDE>(c, 4 * l + 3, p.g[MAT_WD].n_units, n_rows, wd_key);
    if (threadIdx.x == 0) sm.flags[3] = -1;     // ordered by the wait's barrier
    if (!cons_wait(c, ctr + ctr_stage(l, 2), N)) return;
    {
      const MatGeom& g = p.g[MAT_WD];
      const int Kc = g.Ku * 16;
      run_stage<WT, WIDE, true>(
          c, call, sp_wd, Kc, wd_key,
          [&](int u, int, int) {
            const int kc = u / g.n_mb;
            if (sm.flags[3] != kc) {
              const float* m = p.mbuf + (size_t)kc * Kc;
              prep_operand<WT, WIDE>(c, n_rows, Kc, 0, Kc, nullptr, false,
                               [&](int n, int k, auto w) { return ld_global_v<decltype(w)::value>(m + (size_t)n * F + k); });
              if (threadIdx.x == 0) sm.flags[3] = kc;
            }
          },
          [&](int u, int mi, int rr0, int n, float4 v) {
            const int row = (u % g.n_mb) * g.Mu * 16 + mi * 16 + rr0;
            const size_t si = (size_t)l * H + row;
            red_add_f32x4(p.x + (size_t)n * H + row,
                          make_float4(v.x * wscale<WT>(p.s_wd, si), v.y * wscale<WT>(p.s_wd, si + 1),
                                      v.z * wscale<WT>(p.s_wd, si + 2), v.w * wscale<WT>(p.s_wd, si + 3)));
          });
      if (c.abort_) return;
    }
    cons_signal(c, ctr + ctr_stage(l, 3), call, 10 + 4 * (4 * l + 3));
  }

  // ---- S5: final RMSNorm -> verify and draft heads ---------------------------------------
  // Operand column r is packed row r (h before its 1/rms).  LM head P's output for row r at
  // position pos is its verify logits (j = P - pos = 0) or the draft logits of offset j
  // (1 <= j <= K), whose LMH_P b_j term comes from the precomputed bias table.  The call
  // streams the union of the heads its streams need.  The bias depends only on the call's
  // heads and row positions: a single stream with at most kPreUnits head units in this CTA
  // loads its tiles before waiting for the last layer (upper half of `vec`, the gain stays
  // in the lower half); otherwise each chunk stages them once the operand is built.
  g2s_vec(sm.vec, p.final_norm, H);
  const StagePlan sp_head = plan_stage<WT, WIDE>(c, 4 * L, ci->n_heads * p.g[MAT_HEAD].n_units, n_rows, no_key);
  constexpr int kPreUnits = kVecFloats / 2 / (16 * 8);
  const int n_head_units = sp_head.ur.end - sp_head.ur.first;         // contiguous range, step 1
  const bool pre_bias = !WIDE && n_rows <= 8 && H <= kVecFloats / 2 && n_head_units <= kPreUnits;
  float* bias_pre = sm.vec + kVecFloats / 2;                          // [unit][16 rows][8 columns]
  auto head_bias_at = [&](int u, int rr, int n) -> float {
    const MatGeom& g = p.g[MAT_HEAD];
    const int P = ci->heads[u / g.n_units];
    if (n >= n_rows) return 0.f;
    const int j = P - ci->r_pos[n];
    if (j < 1 || j > p.K || ci->r_pos[n] < 1) return 0.f;
    return __ldg(p.head_bias + ((size_t)(P - 1) * p.K + (j - 1)) * p.V + (u % g.n_units) * 16 + rr);
  };
  if (pre_bias)
    for (int o = threadIdx.x; o < n_head_units * 128; o += kConsumerThreads)
      bias_pre[o] = head_bias_at(sp_head.ur.first + (o >> 7), (o >> 3) & 15, o & 7);
  if (!cons_wait(c, ctr + ctr_stage(L - 1, 3), N)) return;
  prep_operand<WT, WIDE>(c, n_rows, H, 0, H, sm.vec, true, from_x);
  {
    const MatGeom& g = p.g[MAT_HEAD];
    float* bias_s = sm.vec;   // [kChunk][16 rows][kMaxCols columns]
    int chunk_u0 = 0;
    run_stage<WT, WIDE>(
        c, call, sp_head, H, no_key,
        [&](int u0, int cnt, int step) {
          chunk_u0 = u0;
          if (pre_bias) return;
          for (int o = threadIdx.x; o < cnt * 16 * kMaxCols; o += kConsumerThreads) {
            const int r = o / (16 * kMaxCols), rr = (o / kMaxCols) & 15, n = o % kMaxCols;
            bias_s[o] = head_bias_at(u0 + r * step, rr, n);
          }
        },
        [&](int u, int mi, int rr, int n, float v, float) {
          const int P = ci->heads[u / g.n_units], pos = ci->r_pos[n], j = P - pos;
          if (pos >= 1 && j >= 0 && j <= p.K) {
            const int id = (u % g.n_units) * g.Mu * 16 + mi * 16 + rr;
            const float b = pre_bias ? bias_pre[((u - sp_head.ur.first) * 16 + rr) * 8 + n]
                                     : bias_s[((u - chunk_u0) * 16 + rr) * kMaxCols + n];
            p.logits[((size_t)(ci->row0 + n) * (kMaxDraft + 1) + j) * p.V + id] =
                v * sm.inv_rms[n] * wscale<WT>(p.s_head, (size_t)(P - 1) * p.V + id) + b;
          }
        });
    if (c.abort_) return;
  }
  cons_signal(c, ctr + ctr_heads(L), call, 10 + 4 * (4 * L));

  // ---- S6: top-k / temperature distribution of every logits row --------------------------
  if (!cons_wait(c, ctr + ctr_heads(L), N)) return;
  timeline(c, call, 1);
  {
    TopkScratch& ts = *reinterpret_cast<TopkScratch*>(sm.act);
    if (ci->emu) {
      // noisy-target pass j = emu (one stream): q = fp32(target logits + sigma N(0,1)) of
      // position pos0 (Box-Muller pairs of purpose 3 + v/2 under the verify round's counters)
      if (blockIdx.x == 0) {
        const int emu = ci->emu, pos0 = ci->st[0].pos0, round = ci->st[0].round;
        const float* lg = p.logits;                                   // row 0, j = 0
        float* zq = p.logits + (size_t)1 * p.V;                        // row 0, slot j = 1
        for (int pr = threadIdx.x; pr < (p.V >> 1); pr += kConsumerThreads) {
          const double2 nz = normal_pair(p.seed, p.stream_ids[0], p.frame_ids[0], round, pos0, pr);
          const float2 l = __ldcg(reinterpret_cast<const float2*>(lg) + pr);
          const float2 z = make_float2((float)((double)l.x + (double)p.sigma * nz.x),
                                       (float)((double)l.y + (double)p.sigma * nz.y));
          reinterpret_cast<float2*>(zq)[pr] = z;
          if (p.trace && round < kMaxCalls) {
            float* dlog = reinterpret_cast<float*>(p.trace + sizeof(mcd_call_trace) * kMaxCalls) +
                          (size_t)kMaxCalls * kMaxRows * p.V;
            reinterpret_cast<float2*>(dlog + ((size_t)round * kMaxRows + (emu - 1)) * p.V)[pr] = z;
          }
        }
        __threadfence();
        consumer_sync();
        block_topk(zq, p.V, p.top_k, p.T, 0, ts, p.draftq + (emu - 1));
        consumer_sync();
      }
    } else {
      // records of call row row0 + r; a tree call keeps every row's records in buffer 0
      const bool tree = WIDE && p.draft_mode == MCD_DRAFT_TREE;
      TopkRec* recs = p.topk + (tree ? 0 : (size_t)(call & 1) * kMaxCols * (kMaxDraft + 1)) +
                      (size_t)ci->row0 * (kMaxDraft + 1);
      const float* lgt = p.logits + (size_t)ci->row0 * (kMaxDraft + 1) * p.V;
      const bool noisy = p.draft_mode == MCD_DRAFT_NOISY_TARGET;
      int pair = 0;
      for (int r = 0; r < n_rows; ++r) {
        const int pos = ci->r_pos[r];
        if (pos < 1) continue;                        // the conditioning row reads no head
        const int kn = noisy ? 0 : min(p.K, p.P - pos);
        for (int j = 0; j <= kn; ++j, ++pair) {
          if (pair % p.n_cta != (int)blockIdx.x) continue;
          const int greedy = (j > 0 && p.draft_mode == MCD_DRAFT_GREEDY) ? 1 : 0;
          block_topk(lgt + ((size_t)r * (kMaxDraft + 1) + j) * p.V, p.V, p.top_k, p.T, greedy, ts,
                     recs + r * (kMaxDraft + 1) + j);
          consumer_sync();
        }
      }
    }
  }
  consumer_sync();
  timeline(c, call, 2);
  timeline_max(c, call, 3);
  // Every CTA's records must be visible before an acceptance step reads them.  One stream:
  // the CTA that arrives last runs its acceptance.  Several: CTA b runs the acceptance of
  // the b-th stream in the call once every CTA has arrived.
  if (threadIdx.x == 0) {
    // release this CTA's records; the last arriver also acquires every earlier arrival's
    // (several streams: the acceptance CTAs acquire through the counter's acquire loads)
    const unsigned old = atom_add_acq_rel(ctr + ctr_topk(L), 1u);
    int mine = -1;
    if (p.S == 1) {
      if (old == N - 1u) mine = 0;
    } else if ((int)blockIdx.x < ci->n_act) {
      if (wait_counter(ctr + ctr_topk(L), N, p.err, p.wait_ns)) mine = ci->act[blockIdx.x];
      else sm.flags[1] = 1;
    }
    sm.flags[2] = mine >= 0 ? 1 : 0;
    sm.flags[4] = mine;
  }
  consumer_sync();
  if (*(volatile int*)&sm.flags[1]) c.abort_ = true;
}


// Acceptance step and next drafts (run by the CTA that finished top-k last).  Every record
// it reads is first staged in shared memory (act + bfrag, 64 KB).
__device__ __noinline__ void accept_step(const FrameParams& p, int call, int s) {
  Smem sm = smem_layout(mcd_dyn_smem);
  const CallInfo* ci = sm.ci;
  const int a = ci->st[s].a, n_d = ci->st[s].n_d, pos0 = ci->st[s].pos0, n_rows = ci->st[s].n_rows;
  const int qrow = ci->st[s].q_row, round = ci->st[s].round, base = ci->base[s];
  const unsigned sid = p.stream_ids[s], fid = p.frame_ids[s];
  const bool noisy = p.draft_mode == MCD_DRAFT_NOISY_TARGET;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const TopkRec* cur = p.topk + (size_t)(call & 1) * kMaxCols * (kMaxDraft + 1);
  const TopkRec* prev = p.topk + (size_t)((call + 1) & 1) * kMaxCols * (kMaxDraft + 1);
  TopkRec* srec = reinterpret_cast<TopkRec*>(sm.act);            // staged records
  const int n_p = (a + 1 + n_d <= p.P) ? n_d + 1 : n_d;
  __shared__ int s_emit[kMaxRows], s_nemit, s_nacc, s_next[kMaxDraft], s_nnext;
  if (s == 0) timeline_p(p, sm.ci, 4, true);
  // p of positions a+1..: this call's verify records (packed rows base + ...); q of the
  // drafts: the previous call's records of its packed row qrow, or the noisy-target passes'
  const int n_pq = n_p + n_d;
  stage_records(srec, n_pq, p.top_k, [&](int r) {
    return r < n_p ? cur + (base + a + 1 + r - pos0) * (kMaxDraft + 1)
                   : (noisy ? p.draftq + (r - n_p) : prev + qrow * (kMaxDraft + 1) + 1 + (r - n_p));
  });
  // The row m whose head drafts the next call is known only after acceptance, so the warps
  // that take no part in it stage every row's draft records meanwhile (if they fit).
  const int idle0 = (n_d + 1) * 32;
  const bool pre = !noisy && idle0 < kConsumerThreads &&
                   (size_t)(n_pq + n_rows * p.K) * sizeof(TopkRec) <= (size_t)(kActBytes + kBfragBytes);
  consumer_sync();
  if (s == 0) timeline_p(p, sm.ci, 5, true);
  // The acceptance rule of every draft in parallel, warp i for draft i (its accept test and
  // the residual draw it would take if it were the first rejection) and warp n_d for the
  // bonus draw; then the chain is read off in order: drafts kept up to the first rejection,
  // whose residual code ends the call, else the bonus code (same decisions as testing the
  // drafts one after another).
  __shared__ int s_ok[kMaxDraft + 1], s_alt[kMaxDraft + 1];
  if (pre)
    stage_records(srec + n_pq, n_rows * p.K, p.top_k,
                  [&](int r) { return cur + (base + r / p.K) * (kMaxDraft + 1) + 1 + r % p.K; }, idle0,
                  kConsumerThreads - idle0);
  if (warp <= n_d) {
    const int i = warp, pos = a + 1 + i;
    if (i < n_d) {
      const TopkRec* pr = srec + i;
      const TopkRec* qr = srec + n_p + i;
      const int d = ci->st[s].drafts[i];
      const unsigned long long wp = warp_weight(pr, d), wq = warp_weight(qr, d);
      const unsigned long long U = uniform_U(p.seed, sid, fid, round, pos, PURPOSE_ACCEPT);
      const bool ok = lt128(mul128x64(mul64(U, wq), pr->S), shl53(wp * qr->S));
      int alt = -1;
      if (!ok) alt = warp_residual(pr, qr, uniform_U(p.seed, sid, fid, round, pos, PURPOSE_TARGET));
      if (lane == 0) {
        s_ok[i] = ok ? 1 : 0;
        s_alt[i] = alt;
      }
    } else if (pos <= p.P) {
      const int b = warp_draw(srec + n_d, uniform_U(p.seed, sid, fid, round, pos, PURPOSE_TARGET));
      if (lane == 0) s_alt[i] = b;
    }
  }
  consumer_sync();
  if (threadIdx.x == 0) {
    int ne = 0, na = 0;
    bool rejected = false;
    for (int i = 0; i < n_d && !rejected; ++i) {
      if (s_ok[i]) {
        s_emit[ne++] = ci->st[s].drafts[i];
        ++na;
      } else {
        s_emit[ne++] = s_alt[i];
        rejected = true;
      }
    }
    if (!rejected && a + 1 + n_d <= p.P) s_emit[ne++] = s_alt[n_d];
    s_nemit = ne;
    s_nacc = na;
  }
  consumer_sync();
  if (s == 0) timeline_p(p, sm.ci, 6, true);
  const int a_new = a + s_nemit;
  const int m = a_new - pos0;
  const int n_next = min(p.K, p.P - a_new);
  // draft records of row m (the row whose head emitted the last code): one warp each (the
  // noisy-target passes that follow draw their drafts themselves)
  if (!noisy) {
    if (!pre) {        // too many rows x drafts to stage up front: row m's records now
      stage_records(srec + n_pq, n_next, p.top_k, [&](int r) { return cur + (base + m) * (kMaxDraft + 1) + 1 + r; });
      consumer_sync();
    }
    const TopkRec* drec = srec + n_pq + (pre ? m * p.K : 0);
    for (int j = 1 + warp; j <= n_next; j += kConsumerWarps) {
      const unsigned long long U = uniform_U(p.seed, sid, fid, round, a_new + j, PURPOSE_DRAFT);
      const int d = warp_draw(drec + (j - 1), U);
      if (lane == 0) s_next[j - 1] = d;
    }
    consumer_sync();
  }
  if (threadIdx.x == 0) {
    s_nnext = n_next;
    DevState* st = p.st + s;
    int* codes_out = p.codes_out ? p.codes_out + (size_t)s * p.P : nullptr;
    for (int t = 0; t < s_nemit; ++t) {
      st->codes[a + 1 + t] = s_emit[t];
      if (codes_out) codes_out[a + t] = s_emit[t];
    }
    if (!noisy)
      for (int j = 0; j < n_next; ++j) st->drafts[j] = s_next[j];
    for (int t = 0; t < s_nemit; ++t) st->emitted_last[t] = s_emit[t];
    const int calls = ci->st[s].calls + 1, heads = ci->st[s].heads_read + ci->phi[s] - ci->plo[s] + 1;
    const int kvr = ci->st[s].kv_rows + pos0 + n_rows, rf = ci->st[s].rows_fed + n_rows;
    const int drafted = ci->st[s].drafted + n_d, accepted = ci->st[s].accepted + s_nacc;
    st->n_emit_last = s_nemit;
    st->n_acc_last = s_nacc;
    st->a = a_new;
    if (noisy && n_next > 0) {           // next: noisy-target pass 1 (row c_a' at position a'+1)
      st->n_d = 0;
      st->pos0 = a_new + 1;
      st->n_rows = 1;
      st->top_pos = a_new + 1;
      st->emu = 1;
      st->emu_n = n_next;
      st->emu_in = s_emit[s_nemit - 1];
    } else {
      st->n_d = n_next;
      st->pos0 = a_new + 1;
      st->n_rows = min(n_next + 1, p.P - a_new);
      st->top_pos = st->pos0 + st->n_rows - 1;
      st->round = round + 1;
    }
    st->first_head_row = 0;
    st->calls = calls;
    st->heads_read = heads;
    st->kv_rows = kvr;
    st->rows_fed = rf;
    st->drafted = drafted;
    st->accepted = accepted;
    st->call = call + 1;
    st->done = a_new >= p.P ? 1 : 0;
    st->q_row = base + m;  // q of the next call's drafts: this call's records of packed row base + m
    if (p.single_call) {
      if (p.emitted_out)
        for (int t = 0; t < s_nemit; ++t) p.emitted_out[t] = s_emit[t];
      if (p.n_emitted_out) *p.n_emitted_out = s_nemit;
    }
    if (a_new >= p.P && p.stats) {
      mcd_frame_stats* fs = p.stats + s;
      fs->calls = calls;
      fs->codes = a_new;
      fs->drafted = drafted;
      fs->accepted = accepted;
      fs->status = 0;
      fs->heads_read = heads;
      fs->kv_rows = kvr;
      fs->rows_fed = rf;
    }
  }
  consumer_sync();
  // optional outputs: trace and stepwise logits
  const int fr = ci->st[s].first_head_row;
  if (p.trace && round < kMaxCalls) {
    uint8_t* tb = p.trace + (size_t)s * p.trace_stride;
    mcd_call_trace* tr = reinterpret_cast<mcd_call_trace*>(tb) + round;
    if (threadIdx.x == 0) {
      tr->a = a;
      tr->n_rows = n_rows;
      tr->pos0 = pos0;
      tr->n_drafts = n_d;
      for (int n = 0; n < kMaxRows; ++n) tr->input_ids[n] = n < n_rows ? ci->r_id[base + n] : -1;
      for (int i = 0; i < kMaxRows; ++i) tr->drafts[i] = i < n_d ? ci->st[s].drafts[i] : -1;
      tr->n_acc = s_nacc;
      tr->n_emit = s_nemit;
      for (int t = 0; t < kMaxRows; ++t) tr->emitted[t] = t < s_nemit ? s_emit[t] : -1;
      tr->n_next = s_nnext;
      for (int j = 0; j < kMaxRows; ++j) tr->next_drafts[j] = (j < s_nnext && !noisy) ? s_next[j] : -1;
      tr->draft_row = m;
    }
    float* vlog = reinterpret_cast<float*>(tb + sizeof(mcd_call_trace) * kMaxCalls);
    float* dlog = vlog + (size_t)kMaxCalls * kMaxRows * p.V;
    for (int idx = threadIdx.x; idx < kMaxRows * p.V; idx += kConsumerThreads) {
      const int n = idx / p.V, v = idx - n * p.V;
      if (n >= fr && n < n_rows)
        vlog[((size_t)round * kMaxRows + n) * p.V + v] =
            __ldcg(p.logits + ((size_t)(base + n) * (kMaxDraft + 1)) * p.V + v);
      if (n < s_nnext && !noisy)
        dlog[((size_t)round * kMaxRows + n) * p.V + v] =
            __ldcg(p.logits + ((size_t)(base + m) * (kMaxDraft + 1) + n + 1) * p.V + v);
    }
  }
  if (p.single_call && p.logits_out) {
    for (int idx = threadIdx.x; idx < (n_rows - fr) * p.V; idx += kConsumerThreads) {
      const int n = fr + idx / p.V, v = idx % p.V;
      p.logits_out[idx] = __ldcg(p.logits + ((size_t)(base + n) * (kMaxDraft + 1)) * p.V + v);
    }
  }
  consumer_sync();
  if (s == 0) timeline_p(p, sm.ci, 7, true);
  if (threadIdx.x == 0) {
    // the last acceptance of the call releases the next call (having acquired the others'
    // state writes through the acceptance counter)
    unsigned* ctr = p.ctr + (size_t)call * p.ctr_stride;
    if (ci->n_act == 1 || atom_add_acq_rel(ctr + ctr_accept(p.L), 1u) == (unsigned)ci->n_act - 1u)
      red_release_add(p.ctr + (size_t)(call + 1) * p.ctr_stride + ctr_ready(p.L), 1u);
  }
}

// Acceptance step of a tree call (one stream; run by the CTA that finished top-k last).
// One warp walks the tree from the first row: the children of the current node are tested
// in rank order, test i keeping its candidate x iff U * S' < 2^53 * W_x, S' being the
// node's weight sum without the candidates rejected so far (one-hot draft distributions);
// a kept child continues the walk, otherwise a code is drawn from the remainder (purpose 0)
// and the call ends.  Then: the next call's candidates (the top-m ids by logit of each
// draft distribution of the last visited row), the kept nodes' K / V moved to their
// positions, the state update, the trace and the release of the next call.
__device__ __noinline__ void accept_tree(const FrameParams& p, int call) {
  Smem sm = smem_layout(mcd_dyn_smem);
  const CallInfo* ci = sm.ci;
  const DevState& st0 = ci->st[0];
  const int a = st0.a, pos0 = st0.pos0, n_rows = st0.n_rows, round = st0.round;
  const unsigned sid = p.stream_ids[0], fid = p.frame_ids[0];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const TopkRec* cur = p.topk;                       // every row's records, buffer 0
  __shared__ int t_emit[kMaxDraft + 1], t_path[kMaxDraft + 1], t_path_row[kMaxDraft + 1], t_res[4];
  __shared__ int t_next[kMaxDraft][kMaxTreeRank];
  if (warp == 0) {
    int node = -1, row = st0.first_head_row, n_emit = 0, plen = 0, tests = 0;
    while (true) {
      const int s = a + 1 + plen;                     // code position of the node's children
      const TopkRec* pr = cur + (size_t)row * (kMaxDraft + 1);
      unsigned long long S_rem = pr->S;
      int rej[kMaxTreeRank];
      int n_rej = 0, kept = -1, kx = -1;
      if (pos0 > 0) {
        for (int r = 0; r < kMaxTreeRank && kept < 0; ++r) {
          int ch = -1;
          for (int k = 0; k < p.tree_n; ++k)
            if (p.tree_parent[k] == node && p.tree_rank[k] == r) ch = k;
          if (ch < 0 || a + p.tree_depth[ch] > p.P) continue;
          const int x = ci->tcand[p.tree_depth[ch] - 1][r];
          const unsigned long long W = warp_weight(pr, x);
          const uint32_t purpose = n_rej == 0 ? (uint32_t)PURPOSE_ACCEPT : kPurposeSibling + (uint32_t)n_rej;
          const unsigned long long U = uniform_U(p.seed, sid, fid, round, s, purpose);
          ++tests;
          if (W > 0 && lt128(mul64(U, S_rem), shl53(W))) {
            kept = ch;
            kx = x;
          } else {
            rej[n_rej++] = x;
            S_rem -= W;
          }
        }
      }
      if (kept >= 0) {
        // rows are the first nodes in tree order: node i was fed at row i + 1 if it exists
        const int kr = kept + 1 < n_rows ? kept + 1 : -1;
        if (lane == 0) {
          t_emit[n_emit] = kx;
          t_path[plen] = kept;
          t_path_row[plen] = kr;
        }
        ++n_emit;
        ++plen;
        if (s == p.P || kr < 0) break;                // the last position: nothing follows
        node = kept;
        row = kr;
        continue;
      }
      if (s <= p.P) {
        const int x = warp_draw_excluding(pr, rej, n_rej, S_rem, uniform_U(p.seed, sid, fid, round, s, PURPOSE_TARGET));
        if (lane == 0) t_emit[n_emit] = x;
        ++n_emit;
      }
      break;
    }
    if (lane == 0) {
      t_res[0] = n_emit;
      t_res[1] = plen;
      t_res[2] = row;
      t_res[3] = tests;
    }
  }
  consumer_sync();
  const int n_emit = t_res[0], plen = t_res[1], drow = t_res[2];
  const int a_new = a + n_emit, n_next = min(p.tree_maxd, p.P - a_new);
  // next candidates: warp j - 1 ranks the draft distribution of depth j of row drow (the
  // record's ids with their fp32 logits; largest logit first, ties to the lower id)
  for (int j = 1 + warp; j <= n_next; j += kConsumerWarps) {
    const TopkRec* dr = cur + (size_t)drow * (kMaxDraft + 1) + j;
    const float* lg = p.logits + ((size_t)drow * (kMaxDraft + 1) + j) * p.V;
    unsigned long long key[kDrawPerLane];
#pragma unroll
    for (int e = 0; e < kDrawPerLane; ++e) {
      const int i = lane * kDrawPerLane + e;
      key[e] = 0ull;
      if (i < dr->n) {
        const int id = dr->ids[i];
        key[e] = ((unsigned long long)f32_key(__ldcg(lg + id)) << 32) | (0xFFFFFFFFu - (uint32_t)id);
      }
    }
    for (int r = 0; r < p.tree_m[j - 1]; ++r) {
      unsigned long long best = 0ull;
#pragma unroll
      for (int e = 0; e < kDrawPerLane; ++e) best = key[e] > best ? key[e] : best;
#pragma unroll
      for (int off = 16; off; off >>= 1) {
        const unsigned long long o = __shfl_xor_sync(0xFFFFFFFFu, best, off);
        best = o > best ? o : best;
      }
#pragma unroll
      for (int e = 0; e < kDrawPerLane; ++e)
        if (key[e] == best) key[e] = 0ull;
      if (lane == 0) t_next[j - 1][r] = best ? (int)(0xFFFFFFFFu - (uint32_t)(best & 0xFFFFFFFFull)) : -1;
    }
  }
  // the kept nodes' keys and values: slot kMaxPos + row -> position a + 2 + t
  {
    int n_mv = 0;
    for (int t = 0; t < plen; ++t) n_mv += t_path_row[t] >= 0 ? 1 : 0;
    const int D4 = p.D >> 2, per = p.L * p.NKV * n_mv * D4;
    for (int i = threadIdx.x; i < 2 * per; i += kConsumerThreads) {
      const bool isv = i >= per;
      const int k = isv ? i - per : i;
      const int d4 = k % D4, t = (k / D4) % n_mv, lg = k / (D4 * n_mv);   // lg = layer * NKV + kv head
      float* base = (isv ? p.vcache : p.kcache) + (size_t)lg * p.kv_slots * p.D;
      const float4 v = __ldcg(reinterpret_cast<const float4*>(base + (size_t)(kMaxPos + t_path_row[t]) * p.D) + d4);
      reinterpret_cast<float4*>(base + (size_t)(a + 2 + t) * p.D)[d4] = v;
    }
  }
  consumer_sync();
  // state of the next call
  __shared__ int t_nvalid, t_maxd;
  if (threadIdx.x == 0) {
    int nv = 0, md = 0;
    for (int i = 0; i < p.tree_n; ++i) {
      const int d = p.tree_depth[i];
      if (d <= n_next && a_new + d < p.P) {
        ++nv;
        md = max(md, d);
      }
    }
    t_nvalid = nv;
    t_maxd = md;
    DevState* st = p.st;
    int* codes_out = p.codes_out;
    for (int t = 0; t < n_emit; ++t) {
      st->codes[a + 1 + t] = t_emit[t];
      if (codes_out) codes_out[a + t] = t_emit[t];
      st->emitted_last[t] = t_emit[t];
    }
    const int calls = st0.calls + 1, heads = st0.heads_read + ci->phi[0] - ci->plo[0] + 1;   // + the last pass
    const int kvr = st0.kv_rows + pos0 + n_rows, rf = st0.rows_fed + n_rows;
    const int drafted = st0.drafted + t_res[3], accepted = st0.accepted + plen;
    st->n_emit_last = n_emit;
    st->n_acc_last = plen;
    st->a = a_new;
    st->n_d = n_next;
    st->pos0 = a_new + 1;
    st->n_rows = 1 + nv;
    st->top_pos = a_new + 1 + md;
    st->round = round + 1;
    st->tpass = 0;
    st->first_head_row = 0;
    st->calls = calls;
    st->heads_read = heads;
    st->kv_rows = kvr;
    st->rows_fed = rf;
    st->drafted = drafted;
    st->accepted = accepted;
    st->call = call + 1;
    st->done = a_new >= p.P ? 1 : 0;
    if (a_new >= p.P && p.stats) {
      mcd_frame_stats* fs = p.stats;
      fs->calls = calls;
      fs->codes = a_new;
      fs->drafted = drafted;
      fs->accepted = accepted;
      fs->status = 0;
      fs->heads_read = heads;
      fs->kv_rows = kvr;
      fs->rows_fed = rf;
    }
  }
  for (int i = threadIdx.x; i < kMaxDraft * kMaxTreeRank; i += kConsumerThreads) {
    const int d = i / kMaxTreeRank, r = i % kMaxTreeRank;
    p.tree_cand[i] = (d < n_next && r < p.tree_m[d]) ? t_next[d][r] : -1;
  }
  consumer_sync();
  // optional trace: the chain record, the draft row's logits, the tree record and every row's
  // verify logits
  if (p.trace && round < kMaxCalls) {
    uint8_t* tb = p.trace;
    mcd_call_trace* tr = reinterpret_cast<mcd_call_trace*>(tb) + round;
    float* dlog = reinterpret_cast<float*>(tb + sizeof(mcd_call_trace) * kMaxCalls) +
                  (size_t)kMaxCalls * kMaxRows * p.V;
    const size_t chain_bytes = sizeof(mcd_call_trace) * kMaxCalls + (size_t)2 * kMaxCalls * kMaxRows * p.V * 4;
    mcd_tree_trace* tt = reinterpret_cast<mcd_tree_trace*>(tb + chain_bytes) + round;
    float* vall = reinterpret_cast<float*>(tb + chain_bytes + sizeof(mcd_tree_trace) * kMaxCalls);
    if (threadIdx.x == 0) {
      tr->a = a;
      tr->n_rows = n_rows;
      tr->pos0 = pos0;
      tr->n_drafts = t_res[3];
      // code fed at call row n: the first call is one pass of plain rows; a tree call feeds
      // c_a, then node n - 1's candidate
      auto row_id = [&](int n) {
        if (n >= n_rows) return -1;
        if (pos0 == 0) return ci->r_id[n];
        if (n == 0) return st0.codes[a];
        return ci->tcand[p.tree_depth[n - 1] - 1][p.tree_rank[n - 1]];
      };
      for (int n = 0; n < kMaxRows; ++n) tr->input_ids[n] = row_id(n);
      for (int i = 0; i < kMaxRows; ++i) tr->drafts[i] = -1;
      tr->n_acc = plen;
      tr->n_emit = n_emit;
      for (int t = 0; t < kMaxRows; ++t) tr->emitted[t] = t < n_emit ? t_emit[t] : -1;
      tr->n_next = n_next;
      for (int j = 0; j < kMaxRows; ++j) tr->next_drafts[j] = j < n_next ? t_next[j][0] : -1;
      tr->draft_row = drow;
      tt->n_rows = n_rows;
      for (int n = 0; n < kMaxTreeRows; ++n) {
        tt->row_node[n] = n >= n_rows ? -1 : pos0 == 0 ? ci->r_node[n] : n - 1;
        tt->row_id[n] = row_id(n);
      }
      tt->n_passes = (n_rows + kMaxCols - 1) / kMaxCols;
      tt->path_len = plen;
      for (int t = 0; t < kMaxDraft + 1; ++t) tt->path[t] = t < plen ? t_path[t] : -1;
      tt->draft_row = drow;
      tt->n_next = n_next;
      for (int d = 0; d < kMaxDraft + 1; ++d)
        for (int r = 0; r < kMaxTreeRank; ++r)
          tt->next_cand[d][r] = (d < n_next && d < kMaxDraft && r < p.tree_m[d]) ? t_next[d][r] : -1;
    }
    for (int idx = threadIdx.x; idx < kMaxTreeRows * p.V; idx += kConsumerThreads) {
      const int n = idx / p.V, v = idx - n * p.V;
      if (n < n_rows && (pos0 > 0 || n > 0))                  // the conditioning row reads no head
        vall[((size_t)round * kMaxTreeRows + n) * p.V + v] =
            __ldcg(p.logits + ((size_t)n * (kMaxDraft + 1)) * p.V + v);
      if (n < n_next)
        dlog[((size_t)round * kMaxRows + n) * p.V + v] =
            __ldcg(p.logits + ((size_t)drow * (kMaxDraft + 1) + n + 1) * p.V + v);
    }
  }
  consumer_sync();
  if (threadIdx.x == 0) red_release_add(p.ctr + (size_t)(call + 1) * p.ctr_stride + ctr_ready(p.L), 1u);
}

// End of a tree call's pass that another pass follows (run by the CTA that finished top-k
// last): its rows' records and K / V stay in place; the next slot runs the next pass.
__device__ __noinline__ void tree_pass_step(const FrameParams& p, int call) {
  Smem sm = smem_layout(mcd_dyn_smem);
  const CallInfo* ci = sm.ci;
  if (threadIdx.x == 0) {
    DevState* st = p.st;
    st->tpass = ci->st[0].tpass + 1;
    st->heads_read = ci->st[0].heads_read + ci->phi[0] - ci->plo[0] + 1;
    st->call = call + 1;
    red_release_add(p.ctr + (size_t)(call + 1) * p.ctr_stride + ctr_ready(p.L), 1u);
  }
}

// Draft step of noisy-target pass j (run by the CTA that finished top-k last): draw the
// draft of position pos0 from the pass's noisy distribution with the draft-purpose uniform
// of the verify round, then set up pass j+1 or, after the last pass, the verify call.
__device__ __noinline__ void emu_step(const FrameParams& p, int call) {
  Smem sm = smem_layout(mcd_dyn_smem);
  const CallInfo* ci = sm.ci;
  const int j = ci->emu, n = ci->st[0].emu_n, round = ci->st[0].round, pos0 = ci->st[0].pos0, a = ci->st[0].a;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  TopkRec* srec = reinterpret_cast<TopkRec*>(sm.act);
  __shared__ int s_d;
  stage_records(srec, 1, p.top_k, [&](int) { return p.draftq + (j - 1); });
  consumer_sync();
  if (warp == 0) {
    const unsigned long long U = uniform_U(p.seed, p.stream_ids[0], p.frame_ids[0], round, pos0, PURPOSE_DRAFT);
    const int d = warp_draw(srec, U);
    if (lane == 0) s_d = d;
  }
  consumer_sync();
  if (threadIdx.x == 0) {
    DevState* st = p.st;
    const int d = s_d;
    st->drafts[j - 1] = d;
    if (j < n) {
      st->emu = j + 1;
      st->emu_in = d;
      st->pos0 = pos0 + 1;
      st->n_rows = 1;
      st->top_pos = pos0 + 1;
    } else {
      st->emu = 0;
      st->emu_n = 0;
      st->n_d = n;
      st->pos0 = a + 1;
      st->n_rows = min(n + 1, p.P - a);
      st->top_pos = st->pos0 + st->n_rows - 1;
      st->round = round + 1;
    }
    st->call = call + 1;
    if (p.trace && round < kMaxCalls) reinterpret_cast<mcd_call_trace*>(p.trace)[round].next_drafts[j - 1] = d;
    red_release_add(p.ctr + (size_t)(call + 1) * p.ctr_stride + ctr_ready(p.L), 1u);
  }
}

template <bool WIDE>
__device__ __forceinline__ bool read_call_state(Cons& c, int call, bool first) {
  const FrameParams& p = c.p;
  Smem& sm = c.sm;
  if (!first) {
    if (!cons_wait(c, p.ctr + (size_t)call * p.ctr_stride + ctr_ready(p.L), 1u)) return false;
  }
  // one parallel read of every stream's state straight into the call snapshot
  constexpr int kWords = sizeof(DevState) / 4;
  CallInfo* ci = sm.ci;
  int* stw = reinterpret_cast<int*>(ci->st);
  for (int i = threadIdx.x; i < p.S * kWords; i += kConsumerThreads)
    stw[i] = __ldcg(reinterpret_cast<const int*>(p.st) + i);
  const bool tree_mode = WIDE && p.draft_mode == MCD_DRAFT_TREE;    // tree calls run wide
  if (tree_mode)
    for (int i = threadIdx.x; i < kMaxDraft * kMaxTreeRank; i += kConsumerThreads)
      ci->tcand[i / kMaxTreeRank][i % kMaxTreeRank] = __ldcg(p.tree_cand + i);
  consumer_sync();
  const DevState* sts = ci->st;
  // a tree call (after the first call): row 0 feeds c_a, then the nodes whose candidates
  // exist and whose code position a + depth < P, in tree order
  const bool tree_rows = tree_mode && sts[0].pos0 > 0 && !sts[0].done;
  // packing order, row bases and the union of heads (one thread)
  if (threadIdx.x == 0) {
    ci->call = call;
    ci->emu = sts[0].emu;
    ci->round0 = sts[0].round;
    int M = 0, n_act = 0;
    unsigned mask = 0;
    for (int s = 0; s < p.S; ++s) {
      ci->base[s] = M;
      if (sts[s].done) continue;
      ci->act[n_act++] = s;
      M = min(M + sts[s].n_rows, kMaxCols);
      int lo, hi;
      head_range(p, sts[s].a, sts[s].top_pos, sts[s].emu, lo, hi);
      ci->plo[s] = lo;
      ci->phi[s] = hi;
      mask |= (hi >= lo) ? ((2u << hi) - (1u << lo)) : 0u;     // bits lo..hi
    }
    ci->M = M;
    ci->n_act = n_act;
    ci->all_done = n_act == 0;
    int nh = 0;
    while (mask) {
      ci->heads[nh++] = __ffs(mask) - 1;
      mask &= mask - 1;
    }
    ci->n_heads = nh;
    ci->row0 = 0;
    ci->tree_more = 0;
    ci->n_tg = 0;
    if (tree_rows) {
      // the call's rows: c_a, then the nodes of depth <= min(n_d, P - 1 - a), a prefix of the
      // breadth-first node list (node i at row i + 1); pass t feeds rows 32 t .. 32 t + 31
      const DevState& st = sts[0];
      int R = 1;
      while (R <= p.tree_n && p.tree_depth[R - 1] <= st.n_d && st.a + p.tree_depth[R - 1] < p.P) ++R;
      const int row0 = st.tpass * kMaxCols, Mp = max(0, min(R - row0, kMaxCols));
      if (R != st.n_rows || Mp == 0) atomicCAS(p.err, 0, (int)MCD_ERR_STATE);   // the acceptance step counted otherwise
      ci->row0 = row0;
      ci->M = Mp;
      ci->tree_more = row0 + Mp < R ? 1 : 0;
      for (int n = 0; n < Mp; ++n) {
        const int m = row0 + n;
        if (m == 0) {
          ci->r_pos[n] = st.pos0;
          ci->r_id[n] = st.codes[st.a];
          ci->r_node[n] = -1;
        } else {
          const int d = p.tree_depth[m - 1];
          ci->r_pos[n] = st.pos0 + d;
          ci->r_id[n] = ci->tcand[d - 1][p.tree_rank[m - 1]];
          ci->r_node[n] = (signed char)(m - 1);
        }
      }
      // attention groups: up to G consecutive rows whose keys (the committed prefix, row 0
      // and the union of their ancestor-or-self sets) fit one task; G spreads the
      // (query head, group) tasks over the CTAs (at most 8 rows, the task's query capacity)
      const int want = max(1, p.n_cta / p.NH);                    // groups per query head
      const int G = min(8, max(1, (Mp + want - 1) / want));
      int ng = 0, r = 0;
      while (r < Mp) {
        const int start = r;
        unsigned long long U = 0ull;
        while (r < Mp && r - start < G) {
          const int m = row0 + r;
          const unsigned long long am = m > 0 ? p.tree_anc[m - 1] : 0ull;
          if (r > start && st.pos0 + 1 + __popcll(U | am) > kTreeKeys) break;
          U |= am;
          ++r;
        }
        ci->tg[ng++] = (signed char)start;
      }
      ci->tg[ng] = (signed char)Mp;
      ci->n_tg = ng;
    }
  }
  consumer_sync();
  // (3) one thread per packed row: stream, position, code fed, layer-0 input row
  if (threadIdx.x < ci->M) {
    const int r = threadIdx.x;
    int s = 0;
    for (int i = 0; i < ci->n_act; ++i)
      if (ci->base[ci->act[i]] <= r) s = ci->act[i];
    const DevState* st = sts + s;
    const int n = r - ci->base[s];
    int pos, id;
    if (tree_rows) {
      pos = ci->r_pos[r];
      id = ci->r_id[r];
    } else {
      pos = st->pos0 + n;
      id = st->emu ? st->emu_in
                   : st->pos0 == 0 ? (n == 0 ? -1 : st->codes[0]) : (n == 0 ? st->codes[st->a] : st->drafts[n - 1]);
      ci->r_anc[r] = (2u << n) - 1u;          // rows 0..n (n <= 31; 2 << 31 wraps to 0)
      ci->r_node[r] = -1;
    }
    // layer-0 input row: cond (position 0), the c0 embedding vector (position 1 without a
    // c0 table), else row `id` of table pos - 1
    if (pos == 0 || (pos == 1 && p.C0V == 0)) {
      ci->r_src[r] = reinterpret_cast<const uint8_t*>((pos == 0 ? p.cond : p.c0emb) + (size_t)s * p.H);
      ci->r_f32[r] = 1;
    } else {
      const int table = pos - 1;
      if (id < 0 || id >= (table == 0 ? p.C0V : p.V)) {   // a c0 outside table 0: fail the frame
        atomicCAS(p.err, 0, (int)MCD_ERR_INVALID_ARG);
        id = 0;
      }
      const int es = p.wdtype == MCD_WEIGHT_F32 ? 4 : 2;      // embedding tables: bf16 unless fp32
      ci->r_src[r] = p.embed + (long long)table * p.embed_stride + (long long)id * p.H * es;
      ci->r_f32[r] = p.wdtype == MCD_WEIGHT_F32 ? 1 : 0;
    }
    ci->r_s[r] = s;
    ci->r_n[r] = n;
    ci->r_pos[r] = pos;
    ci->r_id[r] = id;
  }
  consumer_sync();
  timeline(c, call, 0);
  return true;
}

template <int WT, bool WIDE>
__global__ void __launch_bounds__(kThreads, 1) frame_kernel(const __grid_constant__ FrameParams p) {
  Smem sm = smem_layout(mcd_dyn_smem);
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
  const int call0 = __ldcg(&p.st->call);
  if (warp == kConsumerWarps) {
    if ((tid & 31) == 0) producer_loop(p, sm, call0);
  } else {
    Cons c(p, sm);
    for (int call = call0; call < kMaxSlots; ++call) {
      if (!read_call_state<WIDE>(c, call, call == call0)) break;
      if (sm.ci->all_done) break;
      // a stepwise launch runs one verify call and the noisy-target passes that follow it
      if (p.single_call && call != call0 && !sm.ci->emu) break;
      run_call<WT, WIDE>(c, call);
      if (c.abort_) break;
      if (sm.flags[2]) {
        if (sm.ci->emu)
          emu_step(p, call);
        else if (WIDE && p.draft_mode == MCD_DRAFT_TREE && sm.ci->tree_more)
          tree_pass_step(p, call);
        else if (WIDE && p.draft_mode == MCD_DRAFT_TREE)
          accept_tree(p, call);
        else
          accept_step(p, call, sm.flags[4]);
      }
    }
    if (tid == 0) sm.flags[0] = 1;  // stop the producer
  }
  __syncthreads();
  if (tid == 0 && *(volatile int*)p.err != 0 && p.stats)
    for (int s = 0; s < p.S; ++s) p.stats[s].status = *(volatile int*)p.err;
}

// host-side launcher ------------------------------------------------------------------
// WIDE: the call may pack more than 8 rows (several streams), so the operand has up to 4
// n-tiles; the narrow instantiation serves single-stream decoding.
template <int WT, bool WIDE>
static void* frame_entry() {
  return (void*)frame_kernel<WT, WIDE>;
}

static void* frame_fn(int wdtype, bool wide) {
  switch (wdtype) {
    case MCD_WEIGHT_BF16: return wide ? frame_entry<MCD_WEIGHT_BF16, true>() : frame_entry<MCD_WEIGHT_BF16, false>();
    case MCD_WEIGHT_INT8: return wide ? frame_entry<MCD_WEIGHT_INT8, true>() : frame_entry<MCD_WEIGHT_INT8, false>();
    default: return wide ? frame_entry<MCD_WEIGHT_F32, true>() : frame_entry<MCD_WEIGHT_F32, false>();
  }
}

cudaError_t launch_frame_kernel(const FrameParams& p, cudaStream_t stream) {
  void* args[] = {const_cast<FrameParams*>(&p)};
  const bool wide = p.S * max(p.K + 1, 2) > kMaxRows || p.draft_mode == MCD_DRAFT_TREE;
  return cudaLaunchCooperativeKernel(frame_fn(p.wdtype, wide), dim3(p.n_cta), dim3(kThreads), args, (size_t)kSmemBytes,
                                     stream);
}

cudaError_t prepare_frame_kernel(int* max_ctas_per_sm) {
  for (int wd : {MCD_WEIGHT_F32, MCD_WEIGHT_BF16, MCD_WEIGHT_INT8})
    for (bool wide : {false, true}) {
      cudaError_t e = cudaFuncSetAttribute(frame_fn(wd, wide), cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
      if (e != cudaSuccess) return e;
    }
  return cudaOccupancyMaxActiveBlocksPerMultiprocessor(max_ctas_per_sm, frame_fn(MCD_WEIGHT_BF16, false), kThreads,
                                                       kSmemBytes);
}

int frame_smem_bytes() { return kSmemBytes; }

}  // namespace mcd
