// Top-k / temperature sampling, categorical draw, acceptance test and residual resampling
// on the device (Abstract and Sec. 3.2: the deployed top-k sampling is kept and drafts are
// verified with the standard lossless rule: keep d with probability min(1, p(d)/q(d)),
// otherwise resample from max(0, p - q) renormalised).
//
// A distribution is a list of integer weights (ids in sampling order, W, S = sum W):
//   * top-k set: (fp32 logit desc, id asc); -0 and +0 compare equal; listed by ascending id;
//   * z = fp32 logit / fp32 T; W_i = floor(2^24 * exp32(z_i - z_max)); p(x) = W_x / S;
//   * draw with a 53-bit integer uniform U: first i with U*S < 2^53 * (W_0 + .. + W_i);
//   * accept draft d iff U * Wq_d * S_p < 2^53 * Wp_d * S_q  (u < p(d)/q(d));
//   * residual: N_x = max(0, Wp_x S_q - Wq_x S_p) over p's support in ascending id order,
//     first x with U * R < 2^53 * (N_1 + .. + N_x), R = sum N; R == 0 draws from p.
// Every decision is an exact integer comparison, so a CPU implementation that computes the
// same fp32 exp32 agrees bit for bit; sums are order-free and need no fp64 arithmetic.
#pragma once
#include <cstddef>

#include "mcd_internal.cuh"

namespace mcd {

struct TopkScratch {
  static constexpr int kBins = 256;
  uint32_t hist[kBins];                  // value-range histogram
  uint32_t cand[32];                     // keys of the threshold bin
  uint32_t ncand;
  uint32_t mm[2][kConsumerWarps];        // per-warp maximum / minimum key
  uint32_t part[2][kConsumerWarps][8];   // per-warp counts of the threshold search (double-buffered)
  uint32_t wred[2][kConsumerWarps];      // per-warp maxima / scan totals (double-buffered)
  unsigned long long wsum[kConsumerWarps];
  uint32_t kept_key[kMaxTopK];           // the set in id order: keys and ids
  int kept_id[kMaxTopK];
};
static_assert(sizeof(TopkScratch) <= kActBytes, "top-k scratch must fit the activation region");

// fp32 exponential of d <= 0: Cody-Waite range reduction (Cody and Waite, "Software Manual
// for the Elementary Functions", 1980) with ln 2 = C1 + C2, then e^r by the degree-7 Taylor
// polynomial in Horner form and a scale by 2^n.  Every step is one IEEE single-precision
// operation with round-to-nearest (no contraction into fused multiply-add), constants are
// the fp32 roundings of log2(e), C1 = 0.693359375, C2 = ln 2 - C1 and 1/k!.
__device__ __forceinline__ float exp32_cw(float d) {
  if (d < -87.0f) return 0.0f;
  const float n = rintf(__fmul_rn(d, __int_as_float(0x3fb8aa3b)));
  const float r = __fsub_rn(__fsub_rn(d, __fmul_rn(n, __int_as_float(0x3f318000))),
                            __fmul_rn(n, __int_as_float(0xb95e8083)));
  float p = __int_as_float(0x39500d01);                        // 1/7!
  p = __fadd_rn(__fmul_rn(p, r), __int_as_float(0x3ab60b61));  // 1/6!
  p = __fadd_rn(__fmul_rn(p, r), __int_as_float(0x3c088889));  // 1/5!
  p = __fadd_rn(__fmul_rn(p, r), __int_as_float(0x3d2aaaab));  // 1/4!
  p = __fadd_rn(__fmul_rn(p, r), __int_as_float(0x3e2aaaab));  // 1/3!
  p = __fadd_rn(__fmul_rn(p, r), 0.5f);
  p = __fadd_rn(__fmul_rn(p, r), 1.0f);
  p = __fadd_rn(__fmul_rn(p, r), 1.0f);
  return __fmul_rn(p, __int_as_float(((int)n + 127) << 23));
}

__device__ __forceinline__ uint32_t weight24(float e) { return __float2uint_rd(__fmul_rn(e, 16777216.0f)); }

// ---- exact 128-bit helpers -------------------------------------------------------------
struct U128 {
  unsigned long long lo, hi;
};
__device__ __forceinline__ U128 mul64(unsigned long long a, unsigned long long b) {
  return U128{a * b, __umul64hi(a, b)};
}
// (a * b) for a product known to fit in 128 bits
__device__ __forceinline__ U128 mul128x64(U128 a, unsigned long long b) {
  U128 r = mul64(a.lo, b);
  r.hi += a.hi * b;
  return r;
}
__device__ __forceinline__ U128 shl53(unsigned long long x) { return U128{x << 53, x >> 11}; }
__device__ __forceinline__ bool lt128(U128 a, U128 b) { return a.hi < b.hi || (a.hi == b.hi && a.lo < b.lo); }

__device__ __forceinline__ uint32_t f32_key(float v) {
  uint32_t u = __float_as_uint(v);
  if ((u << 1) == 0u) u = 0u;  // -0 -> +0
  return u ^ ((u >> 31) ? 0xFFFFFFFFu : 0x80000000u);
}
__device__ __forceinline__ float key_f32(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k ^ 0x80000000u) : ~k);
}

// Exclusive scan of v over the 256 consumer threads in thread order; returns the prefix
// and writes the block total to *total.  One barrier (buf selects the scratch half).
__device__ __forceinline__ uint32_t block_exscan(uint32_t v, TopkScratch& s, int buf, uint32_t* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
    if (lane >= o) incl += t;
  }
  if (lane == 31) s.wred[buf][warp] = incl;
  consumer_sync();
  uint32_t before = 0, tot = 0;
#pragma unroll
  for (int w = 0; w < kConsumerWarps; ++w) {
    const uint32_t t = s.wred[buf][w];
    before += (w < warp) ? t : 0u;
    tot += t;
  }
  *total = tot;
  return before + incl - v;
}

// Block-wide (256 consumer threads) top-k of one fp32 row (V % 16 == 0, V <= 4096) into `out`
// (global or shared), listed in ascending id order.  Thread t holds the keys of the E = 4 nj
// consecutive ids E t .. E t + E - 1 (nj = ceil(V / 1024)) in registers, so thread order is id
// order.  Finding the k-th largest key Tk:
//   (1) block maximum and minimum;
//   (2) a 256-bin histogram over the value range [min, max] (bin = trunc((v - min) * 256 /
//       (max - min)), a monotone function of the key, so every bin is an interval of keys);
//   (3) every warp scans the histogram from the top for the bin B holding the k-th largest
//       key; when B holds at most 32 keys they are gathered and one warp ranks them exactly;
//       otherwise (or for a non-finite range) a counting search over key thresholds, 3 bits
//       per step, finds Tk;
//   (4) one prefix scan of the packed per-thread counts (keys > Tk, keys == Tk) places the
//       set in id order (ties at the threshold keep the lowest ids) in shared memory; then
//       thread i computes the weight of entry i (one exponential per thread, not one per key).
// `greedy` replaces the distribution by the one-hot of the argmax (ties: lowest id).  `dbg`,
// when not null, receives clock64() stamps at the phase boundaries (profiling only).
// kJ = float4 chunks per thread the instantiation holds (ceil(V / 1024) <= kJ): block_topk
// runs the smallest instantiation that fits V, so a call executes only the code it needs.
template <int kJ>
static __device__ __noinline__ void block_topk_j(const float* __restrict__ logits, int V, int k, float T, int greedy,
                                                 TopkScratch& s, TopkRec* out, long long* dbg) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
#define MCD_TOPK_STAMP(i) \
  if (dbg && tid == 0) dbg[i] = clock64();
  MCD_TOPK_STAMP(0)
  constexpr int kBins = TopkScratch::kBins;
  static_assert(kBins == kConsumerThreads, "one histogram bin per consumer thread");
  const int nj = (V + 1023) >> 10;                 // float4 chunks per thread
  const int E = 4 * nj;                            // ids per thread
  const int n_valid = max(0, min(E, V - E * tid)); // ids E*tid .. E*tid + n_valid - 1 exist
  uint32_t key[4 * kJ];
#pragma unroll
  for (int j = 0; j < kJ; ++j) {
    const bool ok = 4 * j < n_valid;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    if (ok) v = __ldcg(reinterpret_cast<const float4*>(logits) + (nj * tid + j));
    key[4 * j + 0] = ok ? f32_key(v.x) : 0u;
    key[4 * j + 1] = ok ? f32_key(v.y) : 0u;
    key[4 * j + 2] = ok ? f32_key(v.z) : 0u;
    key[4 * j + 3] = ok ? f32_key(v.w) : 0u;
  }
  uint32_t kmax = 0, kmin = 0xFFFFFFFFu;
#pragma unroll
  for (int e = 0; e < 4 * kJ; ++e) {
    if (e < n_valid) {
      kmax = max(kmax, key[e]);
      kmin = min(kmin, key[e]);
    }
  }
  kmax = __reduce_max_sync(0xFFFFFFFFu, kmax);
  kmin = __reduce_min_sync(0xFFFFFFFFu, kmin);
  if (lane == 0) {
    s.mm[0][warp] = kmax;
    s.mm[1][warp] = kmin;
  }
  s.hist[tid] = 0u;
  if (tid == 0) s.ncand = 0u;
  consumer_sync();
#pragma unroll
  for (int w = 0; w < kConsumerWarps; ++w) {
    kmax = max(kmax, s.mm[0][w]);
    kmin = min(kmin, s.mm[1][w]);
  }
  MCD_TOPK_STAMP(1)
  if (greedy) {
    // argmax, ties to the lowest id (thread order is id order)
    uint32_t best = 0xFFFFFFFFu;
#pragma unroll
    for (int e = 4 * kJ - 1; e >= 0; --e)
      if (e < n_valid && key[e] == kmax) best = (uint32_t)(E * tid + e);
    best = __reduce_min_sync(0xFFFFFFFFu, best);
    if (lane == 0) s.wred[0][warp] = best;
    consumer_sync();
    if (tid == 0) {
      uint32_t b = 0xFFFFFFFFu;
#pragma unroll
      for (int w = 0; w < kConsumerWarps; ++w) b = min(b, s.wred[0][w]);
      out->ids[0] = (int)b;
      out->W[0] = 1u;
      out->S = 1ull;
      out->n = 1;
    }
    MCD_TOPK_STAMP(5)
    return;
  }
  // ---- the k-th largest key -----------------------------------------------------------------
  const float vmin = key_f32(kmin), vmax = key_f32(kmax);
  const float range = __fsub_rn(vmax, vmin);
  const float scale = __fdiv_rn((float)kBins, range);
  const bool binned = isfinite(vmin) && isfinite(vmax) && range > 0.f && isfinite(range) && isfinite(scale);
  auto bin_of = [&](uint32_t kk) {
    return min(kBins - 1, __float2int_rz(__fmul_rn(__fsub_rn(key_f32(kk), vmin), scale)));
  };
  uint32_t Tk = 0;
  bool found = false;
  if (binned) {                                                     // block-uniform
#pragma unroll
    for (int e = 0; e < 4 * kJ; ++e)
      if (e < n_valid) atomicAdd(&s.hist[bin_of(key[e])], 1u);
    consumer_sync();
    // lane L holds bins 8L .. 8L + 7; S(b) = #keys in bins >= b; B = the largest b with S(b) >= k
    uint32_t c8[8];
    {
      const uint4 h0 = reinterpret_cast<const uint4*>(s.hist)[2 * lane];
      const uint4 h1 = reinterpret_cast<const uint4*>(s.hist)[2 * lane + 1];
      c8[0] = h0.x; c8[1] = h0.y; c8[2] = h0.z; c8[3] = h0.w;
      c8[4] = h1.x; c8[5] = h1.y; c8[6] = h1.z; c8[7] = h1.w;
    }
    uint32_t local = 0;
#pragma unroll
    for (int b = 0; b < 8; ++b) local += c8[b];
    uint32_t suf = local;                                // keys in the bins of lanes >= L
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t t = __shfl_down_sync(0xFFFFFFFFu, suf, o);
      if (lane + o < 32) suf += t;
    }
    uint32_t run = suf - local, b_cnt = 0, b_above = 0;
    int b_sel = -1;
#pragma unroll
    for (int b = 7; b >= 0; --b) {
      if (b_sel < 0 && run + c8[b] >= (uint32_t)k) {
        b_sel = 8 * lane + b;
        b_cnt = c8[b];
        b_above = run;
      }
      run += c8[b];
    }
    const unsigned has = __ballot_sync(0xFFFFFFFFu, b_sel >= 0);   // a prefix of the lanes
    const int src = 31 - __clz(has);
    const int B = __shfl_sync(0xFFFFFFFFu, b_sel, src);
    const uint32_t cntB = __shfl_sync(0xFFFFFFFFu, b_cnt, src);
    const uint32_t aboveB = __shfl_sync(0xFFFFFFFFu, b_above, src);
    if (cntB <= 32u) {                                               // block-uniform
#pragma unroll
      for (int e = 0; e < 4 * kJ; ++e)
        if (e < n_valid && bin_of(key[e]) == B) s.cand[atomicAdd(&s.ncand, 1u)] = key[e];
      consumer_sync();
      // the (k - aboveB)-th largest of the bin's keys: gt(i) < need <= ge(i)
      const uint32_t need = (uint32_t)k - aboveB;
      const uint32_t kc = lane < (int)cntB ? s.cand[lane] : 0u;
      uint32_t gt = 0, ge = 0;
      for (int j = 0; j < (int)cntB; ++j) {
        const uint32_t kj = __shfl_sync(0xFFFFFFFFu, kc, j);
        gt += kj > kc ? 1u : 0u;
        ge += kj >= kc ? 1u : 0u;
      }
      const unsigned hit = __ballot_sync(0xFFFFFFFFu, lane < (int)cntB && gt < need && need <= ge);
      Tk = __shfl_sync(0xFFFFFFFFu, kc, __ffs(hit) - 1);
      found = true;
    }
  }
  MCD_TOPK_STAMP(2)
  if (!found) {
    // Counting search.  Invariant: #(key >= lo) >= k > #(key >= hi).  Each step counts 7
    // thresholds splitting [lo, hi) into eighths (one barrier); it stops early when a
    // threshold has exactly k keys at or above it, else when hi = lo + 1.
    uint32_t lo = kmin;
    unsigned long long hi = (unsigned long long)kmax + 1ull;
    int buf = 0;
    while (hi - lo > 1ull) {
      const unsigned long long span = hi - lo;
      uint32_t cnt[7];
#pragma unroll
      for (int i = 0; i < 7; ++i) {
        const uint32_t t = lo + (uint32_t)((span * (unsigned long long)(i + 1)) >> 3);
        uint32_t c = 0;
#pragma unroll
        for (int e = 0; e < 4 * kJ; ++e) c += (e < n_valid && key[e] >= t) ? 1u : 0u;
        cnt[i] = __reduce_add_sync(0xFFFFFFFFu, c);
      }
      if (lane < 7) {
        uint32_t mine = cnt[0];
#pragma unroll
        for (int i = 1; i < 7; ++i) mine = lane == i ? cnt[i] : mine;
        s.part[buf][warp][lane] = mine;
      }
      consumer_sync();
      uint32_t tot = 0;
      if (lane < 7)
#pragma unroll
        for (int w = 0; w < kConsumerWarps; ++w) tot += s.part[buf][w][lane];
      const uint32_t my_t = lo + (uint32_t)((span * (unsigned long long)(lane + 1)) >> 3);
      const unsigned ge = __ballot_sync(0xFFFFFFFFu, lane < 7 && tot >= (uint32_t)k);
      const unsigned eq = __ballot_sync(0xFFFFFFFFu, lane < 7 && tot == (uint32_t)k);
      buf ^= 1;
      if (eq) {
        lo = __shfl_sync(0xFFFFFFFFu, my_t, __ffs(eq) - 1);
        break;
      }
      // thresholds increase with the lane, counts decrease: ge is a prefix of lanes 0..6
      const int nge = __popc(ge);
      const uint32_t new_lo = __shfl_sync(0xFFFFFFFFu, my_t, max(nge - 1, 0));
      const uint32_t new_hi = __shfl_sync(0xFFFFFFFFu, my_t, min(nge, 6));
      if (nge > 0) lo = new_lo;
      if (nge < 7) hi = new_hi;
    }
    Tk = lo;
  }
  MCD_TOPK_STAMP(3)
  // ---- id-ordered compaction with weights: one scan of (keys > Tk) | (keys == Tk) << 16 ------
  uint32_t c_gt = 0, c_eq = 0;
#pragma unroll
  for (int e = 0; e < 4 * kJ; ++e) {
    if (e < n_valid) {
      c_gt += key[e] > Tk ? 1u : 0u;
      c_eq += key[e] == Tk ? 1u : 0u;
    }
  }
  uint32_t tot;
  const uint32_t pre = block_exscan(c_gt | (c_eq << 16), s, 0, &tot);
  const uint32_t krem = (uint32_t)k - (tot & 0xFFFFu);      // threshold keys to keep (>= 1)
  uint32_t tie = pre >> 16;
  uint32_t pos = (pre & 0xFFFFu) + min(tie, krem);
#pragma unroll
  for (int e = 0; e < 4 * kJ; ++e) {
    if (e < n_valid) {
      const uint32_t kv = key[e];
      const bool eq = kv == Tk;
      const bool inc = kv > Tk || (eq && tie < krem);
      tie += eq ? 1u : 0u;
      if (inc) {
        s.kept_key[pos] = kv;
        s.kept_id[pos] = E * tid + e;
        ++pos;
      }
    }
  }
  consumer_sync();
  unsigned long long wsum = 0;
  if (tid < k) {
    const float Td = T;
    const float zmax = __fdiv_rn(key_f32(kmax), Td);
    const float z = __fdiv_rn(key_f32(s.kept_key[tid]), Td);
    const uint32_t w = weight24(exp32_cw(__fsub_rn(z, zmax)));
    out->ids[tid] = s.kept_id[tid];
    out->W[tid] = w;
    wsum = w;
  }
  MCD_TOPK_STAMP(4)
#pragma unroll
  for (int o = 16; o; o >>= 1) wsum += __shfl_xor_sync(0xFFFFFFFFu, wsum, o);
  if (lane == 0) s.wsum[warp] = wsum;
  consumer_sync();
  if (tid == 0) {
    unsigned long long S = 0;
#pragma unroll
    for (int w = 0; w < kConsumerWarps; ++w) S += s.wsum[w];
    out->S = S;
    out->n = k;
  }
  MCD_TOPK_STAMP(5)
#undef MCD_TOPK_STAMP
}
static_assert(kMaxVocab <= 4 * 1024, "block_topk instantiates at most four float4 chunks per thread");
static __device__ __forceinline__ void block_topk(const float* __restrict__ logits, int V, int k, float T, int greedy,
                                                  TopkScratch& s, TopkRec* out, long long* dbg = nullptr) {
  switch ((V + 1023) >> 10) {
    case 1: block_topk_j<1>(logits, V, k, T, greedy, s, out, dbg); break;
    case 2: block_topk_j<2>(logits, V, k, T, greedy, s, out, dbg); break;
    case 3: block_topk_j<3>(logits, V, k, T, greedy, s, out, dbg); break;
    default: block_topk_j<4>(logits, V, k, T, greedy, s, out, dbg); break;
  }
}

// The record helpers read through generic pointers: the frame kernel stages records in
// shared memory, the standalone sampler kernels read the copies their own CTA wrote.

// W_x of a record (0 outside it), evaluated by a full warp (same value on every lane).
__device__ inline __noinline__ uint32_t warp_weight(const TopkRec* r, int x) {
  const int lane = threadIdx.x & 31;
  const int n = r->n;
  int found = -1;
  for (int i = lane; i < n; i += 32)
    if (r->ids[i] == x) found = i;
  const unsigned b = __ballot_sync(0xFFFFFFFFu, found >= 0);
  if (!b) return 0u;
  const int idx = __shfl_sync(0xFFFFFFFFu, found, __ffs(b) - 1);
  return r->W[idx];
}

// Warp-parallel inverse-CDF draw: entry i (0 <= i < n) has value v (lane L holds entries
// 4L..4L+3 in v[0..3]); returns the first i with U * S < 2^53 * (v_0 + ... + v_i).  The
// prefix sums are exact integers, so the result equals the sequential walk's.
constexpr int kDrawPerLane = kMaxTopK / 32;
__device__ inline __noinline__ int warp_draw_lanes(const unsigned long long (&v)[kDrawPerLane], int n,
                                               unsigned long long S, unsigned long long U) {
  const int lane = threadIdx.x & 31;
  unsigned long long tot = 0;
#pragma unroll
  for (int e = 0; e < kDrawPerLane; ++e) tot += v[e];
  unsigned long long incl = tot;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const unsigned long long t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
    if (lane >= o) incl += t;
  }
  unsigned long long c = incl - tot;
  const U128 lhs = mul64(U, S);
  int hit = -1;
#pragma unroll
  for (int e = 0; e < kDrawPerLane; ++e) {
    c += v[e];
    const int i = lane * kDrawPerLane + e;
    if (hit < 0 && i < n && lt128(lhs, shl53(c))) hit = i;
  }
  const unsigned b = __ballot_sync(0xFFFFFFFFu, hit >= 0);
  if (!b) return n - 1;
  return __shfl_sync(0xFFFFFFFFu, hit, __ffs(b) - 1);
}

// Categorical draw from a record, evaluated by a full warp.
__device__ inline __noinline__ int warp_draw(const TopkRec* r, unsigned long long U) {
  const int lane = threadIdx.x & 31, n = r->n;
  unsigned long long v[kDrawPerLane];
#pragma unroll
  for (int e = 0; e < kDrawPerLane; ++e) {
    const int i = lane * kDrawPerLane + e;
    v[e] = i < n ? r->W[i] : 0ull;
  }
  return r->ids[warp_draw_lanes(v, n, r->S, U)];
}

// Draw from p without the ids in ex[0..n_ex) (weights set to zero; S_rem = S minus their
// weights), by a full warp: the residual of one-hot draft distributions tested in turn.
__device__ __forceinline__ int warp_draw_excluding(const TopkRec* r, const int* ex, int n_ex, unsigned long long S_rem,
                                                   unsigned long long U) {
  const int lane = threadIdx.x & 31, n = r->n;
  unsigned long long v[kDrawPerLane];
#pragma unroll
  for (int e = 0; e < kDrawPerLane; ++e) {
    const int i = lane * kDrawPerLane + e;
    v[e] = 0ull;
    if (i < n) {
      const int id = r->ids[i];
      bool out = false;
      for (int t = 0; t < n_ex; ++t) out |= ex[t] == id;
      if (!out) v[e] = r->W[i];
    }
  }
  return r->ids[warp_draw_lanes(v, n, S_rem, U)];
}

// Residual draw from normalise(max(0, p - q)) over p's entries in p's order, by a full warp.
static __device__ __noinline__ int warp_residual(const TopkRec* p, const TopkRec* q, unsigned long long U) {
  const int lane = threadIdx.x & 31;
  const int np = p->n, nq = q->n;
  const unsigned long long Sp = p->S, Sq = q->S;
  int id[kDrawPerLane];
  unsigned long long wq[kDrawPerLane], v[kDrawPerLane];
#pragma unroll
  for (int e = 0; e < kDrawPerLane; ++e) {
    const int i = lane * kDrawPerLane + e;
    id[e] = i < np ? p->ids[i] : -1;
    wq[e] = 0;
  }
  // W_q of each of the lane's ids: binary search of q's ids (records list ascending ids),
  // the lane's searches interleaved
  int lo[kDrawPerLane], hi[kDrawPerLane];
#pragma unroll
  for (int e = 0; e < kDrawPerLane; ++e) {
    lo[e] = 0;
    hi[e] = nq;                          // first index with ids >= id[e] lies in [lo, hi]
  }
  for (int span = nq; span > 0; span >>= 1) {
#pragma unroll
    for (int e = 0; e < kDrawPerLane; ++e) {
      if (lo[e] < hi[e]) {
        const int mid = (lo[e] + hi[e]) >> 1;
        if (q->ids[mid] < id[e]) lo[e] = mid + 1;
        else hi[e] = mid;
      }
    }
  }
#pragma unroll
  for (int e = 0; e < kDrawPerLane; ++e)
    if (id[e] >= 0 && lo[e] < nq && q->ids[lo[e]] == id[e]) wq[e] = q->W[lo[e]];
  unsigned long long R = 0;
#pragma unroll
  for (int e = 0; e < kDrawPerLane; ++e) {
    const int i = lane * kDrawPerLane + e;
    const unsigned long long a = i < np ? (unsigned long long)p->W[i] * Sq : 0ull, b = wq[e] * Sp;
    v[e] = a > b ? a - b : 0ull;
    R += v[e];
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) R += __shfl_xor_sync(0xFFFFFFFFu, R, o);
  if (R == 0) return warp_draw(p, U);
  return p->ids[warp_draw_lanes(v, np, R, U)];
}

struct AcceptResult {
  int n_acc;
  int n_emit;
  int emitted[kMaxRows];
};

// Copy distribution records into shared memory: the header with ids[0..k) and W[0..k) of
// each (k = top_k; entries past a record's n are never read) as 16-byte cp.async chunks, all
// in flight together.  Threads t0 .. t0 + nt - 1 take part; a barrier must follow.
template <class Src>
__device__ __forceinline__ void stage_records(TopkRec* dst, int nrec, int k, Src src, int t0 = 0,
                                              int nt = kConsumerThreads) {
  const int c_ids = (int)((offsetof(TopkRec, ids) + 4 * k + 15) / 16), c_w = (4 * k + 15) / 16;
  const int per = c_ids + c_w, total = nrec * per, me = (int)threadIdx.x - t0;
  if (me < 0 || me >= nt) return;
  for (int i = me; i < total; i += nt) {
    const int r = i / per, ch = i - r * per;
    const int off = ch < c_ids ? ch * 16 : (int)offsetof(TopkRec, W) + (ch - c_ids) * 16;
    cpa16(reinterpret_cast<uint8_t*>(dst + r) + off, reinterpret_cast<const uint8_t*>(src(r)) + off);
  }
  cpa_wait_all();
}
static_assert(sizeof(TopkRec) % 16 == 0 && offsetof(TopkRec, ids) % 16 == 0 && offsetof(TopkRec, W) % 16 == 0,
              "records are copied in 16-byte chunks");

// The acceptance step of one call, evaluated by one full warp.
//   p_row(i): record of the verify distribution of position a+1+i (i = 0..n_d)
//   q_rec(i): draft distribution of draft i (position a+1+i), drafts[i] its id
template <class PRow, class QRec>
__device__ AcceptResult warp_accept(int a, int n_d, int n_pos, const int* drafts, PRow p_row, QRec q_rec,
                                    unsigned long long seed, uint32_t stream, uint32_t frame, int call) {
  AcceptResult res;
  res.n_acc = 0;
  res.n_emit = 0;
  bool rejected = false;
  for (int i = 0; i < n_d && !rejected; ++i) {
    const int s = a + 1 + i;
    const TopkRec* pr = p_row(i);
    const TopkRec* qr = q_rec(i);
    const int d = drafts[i];
    const unsigned long long wp = warp_weight(pr, d), wq = warp_weight(qr, d);
    const unsigned long long U = uniform_U(seed, stream, frame, call, s, PURPOSE_ACCEPT);
    if (lt128(mul128x64(mul64(U, wq), pr->S), shl53(wp * qr->S))) {
      res.emitted[res.n_emit++] = d;
      res.n_acc++;
    } else {
      const unsigned long long U2 = uniform_U(seed, stream, frame, call, s, PURPOSE_TARGET);
      res.emitted[res.n_emit++] = warp_residual(pr, qr, U2);
      rejected = true;
    }
  }
  if (!rejected) {
    const int s = a + 1 + n_d;
    if (s <= n_pos) {
      const unsigned long long U = uniform_U(seed, stream, frame, call, s, PURPOSE_TARGET);
      res.emitted[res.n_emit++] = warp_draw(p_row(n_d), U);
    }
  }
  return res;
}

}  // namespace mcd
