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
#include "mcd_internal.cuh"

namespace mcd {

struct TopkScratch {
  uint32_t part[2][kConsumerWarps][8];   // per-warp counts of the threshold search (double-buffered)
  uint32_t wred[2][kConsumerWarps];      // per-warp maxima / scan totals (double-buffered)
  unsigned long long wsum[kConsumerWarps];
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
// (global or shared), listed in ascending id order.  Thread t holds the keys of ids
// 4t + 1024j + c (j < 4, c < 4) in registers.  The k-th largest key is found by a counting
// search, 3 bits per step (seven thresholds per step, counts reduced with redux.sync, one
// barrier per step); the set is then compacted in id order (ties at the threshold keep the
// lowest ids).  `greedy` replaces the distribution by the one-hot of the argmax.  `dbg`, when
// not null, receives clock64() stamps at the six phase boundaries (profiling only).
static __device__ __forceinline__ void block_topk(const float* __restrict__ logits, int V, int k, float T, int greedy,
                                  TopkScratch& s, TopkRec* out, long long* dbg = nullptr) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
#define MCD_TOPK_STAMP(i) \
  if (dbg && tid == 0) dbg[i] = clock64();
  MCD_TOPK_STAMP(0)
  constexpr int kJ = kMaxVocab / 1024;
  uint32_t key[4 * kJ];
#pragma unroll
  for (int j = 0; j < kJ; ++j) {
    const int i4 = tid + kConsumerThreads * j;
    float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
    const bool ok = 4 * i4 < V;
    if (ok) v = __ldcg(reinterpret_cast<const float4*>(logits) + i4);
    key[4 * j + 0] = ok ? f32_key(v.x) : 0u;   // key 0 (a NaN pattern) is never counted
    key[4 * j + 1] = ok ? f32_key(v.y) : 0u;
    key[4 * j + 2] = ok ? f32_key(v.z) : 0u;
    key[4 * j + 3] = ok ? f32_key(v.w) : 0u;
  }
  // block maximum and minimum (padding keys: 0 never wins the maximum, ~0 never the minimum)
  const int nj = (V + 1023) >> 10;
  uint32_t kmax = 0, kmin = 0xFFFFFFFFu;
#pragma unroll
  for (int e = 0; e < 4 * kJ; ++e) {
    if ((e >> 2) < nj) {
      kmax = max(kmax, key[e]);
      kmin = min(kmin, key[e]);
    }
  }
  kmax = __reduce_max_sync(0xFFFFFFFFu, kmax);
  kmin = __reduce_min_sync(0xFFFFFFFFu, kmin);
  if (lane == 0) {
    s.wred[0][warp] = kmax;
    s.wred[1][warp] = kmin;
  }
  consumer_sync();
#pragma unroll
  for (int w = 0; w < kConsumerWarps; ++w) {
    kmax = max(kmax, s.wred[0][w]);
    kmin = min(kmin, s.wred[1][w]);
  }
  MCD_TOPK_STAMP(1)
  // Counting search for the k-th largest key.  Invariant: #(key >= lo) >= k > #(key >= hi).
  // Each step counts 7 thresholds splitting [lo, hi) into eighths (one barrier); it stops
  // early when a threshold has exactly k keys at or above it (then that set is the answer
  // and no tie needs splitting), else when hi = lo + 1 (lo is the k-th largest key).
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
      for (int e = 0; e < 4 * kJ; ++e)
        if ((e >> 2) < nj) c += key[e] >= t ? 1u : 0u;
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
    if (eq) {                                           // exactly k keys >= that threshold
      lo = __shfl_sync(0xFFFFFFFFu, my_t, __ffs(eq) - 1);
      break;
    }
    // thresholds are increasing in lane, counts decreasing: ge is a prefix of lanes 0..6
    const int nge = __popc(ge);
    const uint32_t new_lo = __shfl_sync(0xFFFFFFFFu, my_t, max(nge - 1, 0));
    const uint32_t new_hi = __shfl_sync(0xFFFFFFFFu, my_t, min(nge, 6));
    if (nge > 0) lo = new_lo;
    if (nge < 7) hi = new_hi;
  }
  const uint32_t Tk = lo;
  MCD_TOPK_STAMP(2)
  // counts above and at the threshold
  uint32_t c_gt = 0, c_eq = 0;
#pragma unroll
  for (int e = 0; e < 4 * kJ; ++e) {
    c_gt += key[e] > Tk ? 1u : 0u;
    c_eq += key[e] == Tk ? 1u : 0u;
  }
  c_gt = __reduce_add_sync(0xFFFFFFFFu, c_gt);
  c_eq = __reduce_add_sync(0xFFFFFFFFu, c_eq);
  if (lane == 0) {
    s.part[buf][warp][0] = c_gt;
    s.part[buf][warp][1] = c_eq;
  }
  consumer_sync();
  uint32_t n_gt = 0, n_eq = 0;
#pragma unroll
  for (int w = 0; w < kConsumerWarps; ++w) {
    n_gt += s.part[buf][w][0];
    n_eq += s.part[buf][w][1];
  }
  const uint32_t krem = (uint32_t)k - n_gt;      // >= 1 threshold keys to keep, lowest ids first
  const bool all_eq = n_eq == krem;
  MCD_TOPK_STAMP(3)
  // id-ordered compaction with weights
  const float Td = T;
  const float zmax = __fdiv_rn(key_f32(kmax), Td);
  uint32_t base = 0, tie_base = 0;
  unsigned long long wsum = 0;
  int sbuf = 1;
#pragma unroll
  for (int j = 0; j < kJ; ++j) {
    if (1024 * j >= V) break;                    // block-uniform
    bool inc[4];
    uint32_t n_inc = 0, n_tie = 0;
#pragma unroll
    for (int c = 0; c < 4; ++c) n_tie += key[4 * j + c] == Tk ? 1u : 0u;
    uint32_t tie_pre = 0;
    if (!all_eq) {
      uint32_t tot;
      tie_pre = tie_base + block_exscan(n_tie, s, sbuf, &tot);
      sbuf ^= 1;
      tie_base += tot;
    }
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const uint32_t kv = key[4 * j + c];
      const bool eq = kv == Tk;
      inc[c] = kv > Tk || (eq && (all_eq || tie_pre < krem));
      tie_pre += eq ? 1u : 0u;
      n_inc += inc[c] ? 1u : 0u;
    }
    uint32_t tot;
    uint32_t pos = base + block_exscan(n_inc, s, sbuf, &tot);
    sbuf ^= 1;
    base += tot;
    if (!greedy) {
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        if (inc[c]) {
          const float z = __fdiv_rn(key_f32(key[4 * j + c]), Td);
          const uint32_t w = weight24(exp32_cw(__fsub_rn(z, zmax)));
          out->ids[pos] = 4 * (tid + kConsumerThreads * j) + c;
          out->W[pos] = w;
          wsum += w;
          ++pos;
        }
      }
    }
  }
  MCD_TOPK_STAMP(4)
  if (greedy) {
    // argmax, ties to the lowest id
    uint32_t best = 0xFFFFFFFFu;
#pragma unroll
    for (int j = 0; j < kJ; ++j)
#pragma unroll
      for (int c = 0; c < 4; ++c) {
        const uint32_t id = 4 * (tid + kConsumerThreads * j) + c;
        if (key[4 * j + c] == kmax && (int)id < V) best = min(best, id);
      }
    best = __reduce_min_sync(0xFFFFFFFFu, best);
    if (lane == 0) s.wred[sbuf][warp] = best;
    consumer_sync();
    if (tid == 0) {
      uint32_t b = 0xFFFFFFFFu;
#pragma unroll
      for (int w = 0; w < kConsumerWarps; ++w) b = min(b, s.wred[sbuf][w]);
      out->ids[0] = (int)b;
      out->W[0] = 1u;
      out->S = 1ull;
      out->n = 1;
    }
  } else {
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
  }
  MCD_TOPK_STAMP(5)
#undef MCD_TOPK_STAMP
}

// The record helpers read through generic pointers: the frame kernel stages records in
// shared memory, the standalone sampler kernels read the copies their own CTA wrote.

// W_x of a record (0 outside it), evaluated by a full warp (same value on every lane).
__device__ __forceinline__ uint32_t warp_weight(const TopkRec* r, int x) {
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
__device__ __forceinline__ int warp_draw_lanes(const unsigned long long (&v)[kDrawPerLane], int n,
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
__device__ __forceinline__ int warp_draw(const TopkRec* r, unsigned long long U) {
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
static __device__ int warp_residual(const TopkRec* p, const TopkRec* q, unsigned long long U) {
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
  for (int j = 0; j < nq; ++j) {       // q's entries broadcast to every lane
    const int qid = q->ids[j];
    const unsigned long long qw = q->W[j];
#pragma unroll
    for (int e = 0; e < kDrawPerLane; ++e)
      if (id[e] == qid) wq[e] = qw;
  }
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
