// Top-k / temperature softmax, categorical draw, acceptance test and residual resampling
// on the device (Abstract and Sec. 3.2: the deployed top-k sampling is kept and drafts are
// verified with the standard lossless rule: keep d with probability min(1, p(d)/q(d)),
// otherwise resample from max(0, p - q) renormalised).
//
// Fixed so that the GPU and the CPU oracle take every integer decision from the same fp32
// logits and the same uniforms:
//   * top-k set and order: (fp32 logit desc, id asc); -0 and +0 compare equal;
//   * z = double(logit) / double(T), e_i = exp(z_i - z_max), S = sequential sum in order;
//   * draw: first i with u*S < e_0 + ... + e_i;
//   * accept: u * q(d) < p(d) with p(x) = e_x / S (0 outside the top-k);
//   * residual: r(x) = max(0, p(x) - q(x)) over p's support in ascending id order, drawn
//     like a categorical with R = sequential sum of r; R == 0 draws from p.
#pragma once
#include "mcd_internal.cuh"

namespace mcd {

struct TopkScratch {
  uint32_t keys[kMaxVocab];
  uint32_t hist[256];
  uint32_t cand_key[kMaxTopK];
  int cand_id[kMaxTopK];
  double e[kMaxTopK];
  int misc[8];
  int warp_tot[kConsumerWarps];
};
static_assert(sizeof(TopkScratch) <= kActBytes, "top-k scratch must fit the activation region");

struct ResidualScratch {
  double r[kMaxTopK];
  int x[kMaxTopK];
};

__device__ __forceinline__ uint32_t f32_key(float v) {
  uint32_t u = __float_as_uint(v);
  if ((u << 1) == 0u) u = 0u;  // -0 -> +0
  return u ^ ((u >> 31) ? 0xFFFFFFFFu : 0x80000000u);
}
__device__ __forceinline__ float key_f32(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k ^ 0x80000000u) : ~k);
}

// Block-wide (256 consumer threads) top-k of one fp32 row.  `greedy` replaces the
// distribution by the one-hot of its first entry.  Result written to `out` (global).
static __device__ void block_topk(const float* __restrict__ logits, int V, int k, float T, int greedy,
                           TopkScratch& s, TopkRec* out) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int i = tid; i < (V >> 2); i += 2 * kConsumerThreads) {   // V % 16 == 0: 16-byte loads, two in flight
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
  if (tid < k) {
    const double Td = (double)T;
    const double m = (double)key_f32(s.cand_key[0]) / Td;
    const double z = (double)key_f32(s.cand_key[tid]) / Td;
    const double e = exp(z - m);
    s.e[tid] = e;
    out->ids[tid] = s.cand_id[tid];
    out->e[tid] = greedy ? (tid == 0 ? 1.0 : 0.0) : e;
  }
  consumer_sync();
  if (tid == 0) {
    double S = 0.0;
    for (int j = 0; j < k; ++j) S += s.e[j];
    out->S = greedy ? 1.0 : S;
    out->n = greedy ? 1 : k;
  }
}

// The helpers below read records through generic pointers: the frame kernel stages them in
// shared memory, the standalone sampler kernels read the global copies their own CTA wrote.

// p(x) of a distribution record, evaluated by a full warp (same value on every lane).
__device__ __forceinline__ double warp_prob(const TopkRec* r, int x) {
  const int lane = threadIdx.x & 31;
  const int n = r->n;
  int found = -1;
  for (int i = lane; i < n; i += 32)
    if (r->ids[i] == x) found = i;
  const unsigned b = __ballot_sync(0xFFFFFFFFu, found >= 0);
  if (!b) return 0.0;
  const int idx = __shfl_sync(0xFFFFFFFFu, found, __ffs(b) - 1);
  return r->e[idx] / r->S;
}

// Sequential inverse-CDF draw (one thread).
__device__ __forceinline__ int seq_draw(const TopkRec* r, double u) {
  const int n = r->n;
  const double t = u * r->S;
  double c = 0.0;
  for (int i = 0; i < n; ++i) {
    c += r->e[i];
    if (t < c) return r->ids[i];
  }
  return r->ids[n - 1];
}

// Residual draw from normalise(max(0, p - q)), evaluated by a full warp.
static __device__ int warp_residual(const TopkRec* p, const TopkRec* q, double u, ResidualScratch& rs) {
  const int lane = threadIdx.x & 31;
  const int np = p->n, nq = q->n;
  const double Sp = p->S, Sq = q->S;
  for (int i = lane; i < np; i += 32) {
    const int x = p->ids[i];
    const double px = p->e[i] / Sp;
    double qx = 0.0;
    for (int j = 0; j < nq; ++j)
      if (q->ids[j] == x) {
        qx = q->e[j] / Sq;
        break;
      }
    int rank = 0;
    for (int j = 0; j < np; ++j) rank += (p->ids[j] < x);
    rs.r[rank] = fmax(0.0, px - qx);
    rs.x[rank] = x;
  }
  __syncwarp();
  int out = 0;
  if (lane == 0) {
    double R = 0.0;
    for (int i = 0; i < np; ++i) R += rs.r[i];
    if (R == 0.0) {
      out = seq_draw(p, u);
    } else {
      const double t = u * R;
      double c = 0.0;
      out = rs.x[np - 1];
      int last = rs.x[np - 1];
      bool hit = false;
      for (int i = 0; i < np && !hit; ++i) {
        c += rs.r[i];
        if (rs.r[i] > 0.0) last = rs.x[i];
        if (t < c) {
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
    const double pd = warp_prob(pr, d);
    const double qd = warp_prob(qr, d);
    const double u = uniform_u(seed, stream, frame, call, s, PURPOSE_ACCEPT);
    if (u * qd < pd) {
      res.emitted[res.n_emit++] = d;
      res.n_acc++;
    } else {
      const double u2 = uniform_u(seed, stream, frame, call, s, PURPOSE_TARGET);
      res.emitted[res.n_emit++] = warp_residual(pr, qr, u2, rs);
      rejected = true;
    }
  }
  if (!rejected) {
    const int s = a + 1 + n_d;
    if (s <= n_pos) {
      const double u = uniform_u(seed, stream, frame, call, s, PURPOSE_TARGET);
      int x = 0;
      if ((threadIdx.x & 31) == 0) x = seq_draw(p_row(n_d), u);
      res.emitted[res.n_emit++] = __shfl_sync(0xFFFFFFFFu, x, 0);
    }
  }
  return res;
}

}  // namespace mcd
