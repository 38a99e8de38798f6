// Top-k / temperature sampling, categorical draw, acceptance test and residual resampling
// on the device (Abstract and Sec. 3.2: the deployed top-k sampling is kept and drafts are
// verified with the standard lossless rule: keep d with probability min(1, p(d)/q(d)),
// otherwise resample from max(0, p - q) renormalised).
//
// A distribution is a list of integer weights (ids in sampling order, W, S = sum W):
//   * top-k set and order: (fp32 logit desc, id asc); -0 and +0 compare equal;
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
  uint32_t keys[kMaxVocab];
  uint32_t hist[256];
  uint32_t cand_key[kMaxTopK];
  int cand_id[kMaxTopK];
  unsigned long long wsum[kConsumerWarps];
  int misc[8];
  int warp_tot[kConsumerWarps];
};
static_assert(sizeof(TopkScratch) <= kActBytes, "top-k scratch must fit the activation region");

struct ResidualScratch {
  unsigned long long n[kMaxTopK];
  int x[kMaxTopK];
};

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

// Block-wide (256 consumer threads) top-k of one fp32 row into `out` (global or shared).
// `greedy` replaces the distribution by the one-hot of its first entry.
static __device__ void block_topk(const float* __restrict__ logits, int V, int k, float T, int greedy,
                                  TopkScratch& s, TopkRec* out) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int i = tid; i < (V >> 2); i += 2 * kConsumerThreads) {   // V % 16 == 0: two 16-byte loads in flight
    const int i2 = i + kConsumerThreads;
    const float4 a = __ldcg(reinterpret_cast<const float4*>(logits) + i);
    float4 b = make_float4(0.f, 0.f, 0.f, 0.f);
    if (i2 < (V >> 2)) b = __ldcg(reinterpret_cast<const float4*>(logits) + i2);
    s.keys[4 * i] = f32_key(a.x);
    s.keys[4 * i + 1] = f32_key(a.y);
    s.keys[4 * i + 2] = f32_key(a.z);
    s.keys[4 * i + 3] = f32_key(a.w);
    if (i2 < (V >> 2)) {
      s.keys[4 * i2] = f32_key(b.x);
      s.keys[4 * i2 + 1] = f32_key(b.y);
      s.keys[4 * i2 + 2] = f32_key(b.z);
      s.keys[4 * i2 + 3] = f32_key(b.w);
    }
  }
  // radix select of the k-th largest key, 8 bits per pass
  uint32_t prefix = 0, mask = 0;
  int krem = k;
  int count_eq = 0;
  for (int pass = 3; pass >= 0; --pass) {
    const int shift = pass * 8;
    s.hist[tid] = 0;
    consumer_sync();
    for (int i = tid; i < V; i += kConsumerThreads) {
      const uint32_t key = s.keys[i];
      if ((key & mask) == prefix) atomicAdd(&s.hist[(key >> shift) & 255u], 1u);
    }
    consumer_sync();
    if (warp == 0) {
      int cnt[8], tot = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        cnt[j] = (int)s.hist[255 - 8 * lane - j];
        tot += cnt[j];
      }
      int incl = tot;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        int n = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += n;
      }
      int c = incl - tot;
      if (c < krem && krem <= c + tot) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (c < krem && krem <= c + cnt[j]) {
            s.misc[0] = 255 - 8 * lane - j;
            s.misc[1] = c;
            s.misc[2] = cnt[j];
          }
          c += cnt[j];
        }
      }
    }
    consumer_sync();
    prefix |= (uint32_t)s.misc[0] << shift;
    mask |= 255u << shift;
    krem -= s.misc[1];
    count_eq = s.misc[2];
    consumer_sync();
  }
  const uint32_t Tk = prefix;
  const int n_gt = k - krem;
  if (tid == 0) {
    s.misc[4] = 0;
    s.misc[5] = 0;
  }
  consumer_sync();
  const bool take_all_eq = (count_eq == krem);
  for (int i = tid; i < V; i += kConsumerThreads) {
    const uint32_t key = s.keys[i];
    if (key > Tk) {
      const int slot = atomicAdd(&s.misc[4], 1);
      s.cand_key[slot] = key;
      s.cand_id[slot] = i;
    } else if (key == Tk && take_all_eq) {
      const int slot = n_gt + atomicAdd(&s.misc[5], 1);
      s.cand_key[slot] = key;
      s.cand_id[slot] = i;
    }
  }
  if (!take_all_eq) {  // the krem lowest ids among the keys equal to the threshold
    int base = 0;
    for (int c0 = 0; c0 < V && base < krem; c0 += kConsumerThreads) {
      const int i = c0 + tid;
      const bool eq = (i < V) && (s.keys[i] == Tk);
      const unsigned bal = __ballot_sync(0xFFFFFFFFu, eq);
      if (lane == 0) s.warp_tot[warp] = __popc(bal);
      consumer_sync();
      int before = 0, total = 0;
#pragma unroll
      for (int w = 0; w < kConsumerWarps; ++w) {
        const int t = s.warp_tot[w];
        before += (w < warp) ? t : 0;
        total += t;
      }
      const int rank = base + before + __popc(bal & ((1u << lane) - 1u));
      if (eq && rank < krem) {
        s.cand_key[n_gt + rank] = Tk;
        s.cand_id[n_gt + rank] = i;
      }
      base += total;
      consumer_sync();
    }
  }
  consumer_sync();
  // rank sort by (key desc, id asc)
  uint32_t mk = 0;
  int mid = 0, rank = 0;
  if (tid < k) {
    mk = s.cand_key[tid];
    mid = s.cand_id[tid];
    for (int j = 0; j < k; ++j) {
      const uint32_t kj = s.cand_key[j];
      const int ij = s.cand_id[j];
      rank += (kj > mk) || (kj == mk && ij < mid);
    }
  }
  consumer_sync();
  if (tid < k) {
    s.cand_key[rank] = mk;
    s.cand_id[rank] = mid;
  }
  consumer_sync();
  // integer weights and their (order-free) sum
  uint32_t w = 0;
  if (tid < k) {
    const float z0 = __fdiv_rn(key_f32(s.cand_key[0]), T);
    const float z = __fdiv_rn(key_f32(s.cand_key[tid]), T);
    w = greedy ? (tid == 0 ? 1u : 0u) : weight24(exp32_cw(__fsub_rn(z, z0)));
    out->ids[tid] = s.cand_id[tid];
    out->W[tid] = w;
  }
  unsigned long long ws = w;
#pragma unroll
  for (int o = 16; o; o >>= 1) ws += __shfl_xor_sync(0xFFFFFFFFu, ws, o);
  if (lane == 0) s.wsum[warp] = ws;
  consumer_sync();
  if (tid == 0) {
    unsigned long long S = 0;
#pragma unroll
    for (int w2 = 0; w2 < kConsumerWarps; ++w2) S += s.wsum[w2];
    out->S = S;
    out->n = greedy ? 1 : k;
  }
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

// Inverse-CDF draw (one thread).
__device__ __forceinline__ int seq_draw(const TopkRec* r, unsigned long long U) {
  const int n = r->n;
  const U128 lhs = mul64(U, r->S);
  unsigned long long c = 0;
  for (int i = 0; i < n; ++i) {
    c += r->W[i];
    if (lt128(lhs, shl53(c))) return r->ids[i];
  }
  return r->ids[n - 1];
}

// Residual draw from normalise(max(0, p - q)), evaluated by a full warp.
static __device__ int warp_residual(const TopkRec* p, const TopkRec* q, unsigned long long U, ResidualScratch& rs) {
  const int lane = threadIdx.x & 31;
  const int np = p->n, nq = q->n;
  const unsigned long long Sp = p->S, Sq = q->S;
  for (int i = lane; i < np; i += 32) {
    const int x = p->ids[i];
    unsigned long long wq = 0;
    for (int j = 0; j < nq; ++j)
      if (q->ids[j] == x) {
        wq = q->W[j];
        break;
      }
    const unsigned long long a = (unsigned long long)p->W[i] * Sq, b = wq * Sp;
    int rank = 0;
    for (int j = 0; j < np; ++j) rank += (p->ids[j] < x);
    rs.n[rank] = a > b ? a - b : 0ull;
    rs.x[rank] = x;
  }
  __syncwarp();
  int out = 0;
  if (lane == 0) {
    unsigned long long R = 0;
    for (int i = 0; i < np; ++i) R += rs.n[i];
    if (R == 0) {
      out = seq_draw(p, U);
    } else {
      const U128 lhs = mul64(U, R);
      unsigned long long c = 0;
      int last = rs.x[np - 1];
      bool hit = false;
      for (int i = 0; i < np && !hit; ++i) {
        c += rs.n[i];
        if (rs.n[i] > 0) last = rs.x[i];
        if (lt128(lhs, shl53(c))) {
          out = rs.x[i];
          hit = true;
        }
      }
      if (!hit) out = last;
    }
  }
  __syncwarp();
  return __shfl_sync(0xFFFFFFFFu, out, 0);
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
                                    unsigned long long seed, uint32_t stream, uint32_t frame, int call,
                                    ResidualScratch& rs) {
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
      res.emitted[res.n_emit++] = warp_residual(pr, qr, U2, rs);
      rejected = true;
    }
  }
  if (!rejected) {
    const int s = a + 1 + n_d;
    if (s <= n_pos) {
      const unsigned long long U = uniform_U(seed, stream, frame, call, s, PURPOSE_TARGET);
      int x = 0;
      if ((threadIdx.x & 31) == 0) x = seq_draw(p_row(n_d), U);
      res.emitted[res.n_emit++] = __shfl_sync(0xFFFFFFFFu, x, 0);
    }
  }
  return res;
}

}  // namespace mcd
