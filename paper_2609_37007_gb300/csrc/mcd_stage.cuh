// Shared machinery of the persistent weight-streaming kernels (the frame kernel of the
// MultiCodeDecoder and the outer CodeDecoder's step kernel): shared-memory layout, the
// unit schedule, the consumer side of the weight ring, the activation operand builder and
// the per-stage unit GEMMs with their batched epilogue.
//
// Work split.  Weight matrices are cut into units of <= 32 KB (see mcd_internal.cuh).
// Unit u of a backbone stage goes to CTA (u + rot) mod n_cta, rot being the number of units
// of all earlier stages, so every CTA streams about the same bytes; the LM-head stage hands
// each CTA a contiguous block of units so that a CTA mostly reads one head.  In each CTA a
// producer warp issues 1-D bulk copies (cp.async.bulk, evict-first) of its units into a
// 4-slot shared-memory ring as fast as slots free up -- across stage and call boundaries --
// while 8 consumer warps wait for the stage's inputs (a global counter reaching n_cta),
// turn the activations into bf16 hi/lo mma operands in one pass from global memory and
// multiply each unit with mma.m16n8k16 (weights as the 16-row A side, up to 8 activation
// columns per n-tile as B).  RMSNorm is applied as a per-column scale in the epilogue:
// W (x . g) / rms.  Every wait is bounded.
#pragma once
#include <type_traits>
#include "mcd_internal.cuh"

namespace mcd {

// Vector width tags of the operand loaders: ld(n, k, Vec2{}) -> float2, Vec4{} -> float4.
using Vec2 = std::integral_constant<int, 2>;
using Vec4 = std::integral_constant<int, 4>;
template <int W> using vecf = typename std::conditional<W == 4, float4, float2>::type;


// Snapshot of one call: the packed rows and every stream's state.
struct CallInfo {
  int call;                    // slot (counter set) of this pass
  int M;                       // packed rows
  int n_act;                   // streams with rows in this call
  int n_heads;                 // LM heads streamed
  int heads[16];               // their positions P
  int emu, round0;             // noisy-target pass flag, stream 0's verify round (S = 1)
  int all_done;
  // packed rows: stream, row within the stream, position, code fed, layer-0 input row
  int r_s[kMaxCols], r_n[kMaxCols], r_pos[kMaxCols], r_id[kMaxCols], r_f32[kMaxCols];
  const uint8_t* r_src[kMaxCols];
  // rows of the same stream visible to packed row r (bit n: the stream's row n): every
  // earlier row and itself, or for a tree call the first row, its ancestors and itself
  unsigned r_anc[kMaxCols];
  signed char r_node[kMaxCols];                  // tree node of the row (-1: none)
  int tcand[kMaxDraft][kMaxTreeRank];            // tree call: candidates of its nodes
  // tree call: the pass feeds rows row0 .. row0 + M - 1 of the call (tree_more: a later pass
  // follows); attention groups g = tg[g] .. tg[g + 1] - 1 (pass rows), n_tg of them
  int row0, tree_more, n_tg;
  signed char tg[kMaxCols + 1];
  // per stream (index = stream): its state and the derived packing
  DevState st[kMaxStreams];
  int act[kMaxStreams];        // active streams in packing order
  int base[kMaxStreams], plo[kMaxStreams], phi[kMaxStreams];
};

struct Smem {
  uint8_t* ring;
  float* act;
  uint8_t* bfrag;
  float* red;
  float* vec;      // the current stage's norm gain
  float* part;     // [kConsumerWarps][kMaxCols] partial sums of squares
  uint64_t* full;
  uint64_t* empty;
  int* flags;      // [0] stop, [1] abort, [2] last-arriver, [3] current head / chunk
  float* inv_rms;  // [kMaxCols]
  CallInfo* ci;    // snapshot of the call's state
};

constexpr int kRingOff = 0;
constexpr int kActOff = kRingOff + kNumSlots * kSlotBytes;
constexpr int kBfragOff = kActOff + kActBytes;
constexpr int kRedOff = kBfragOff + kBfragBytes;
constexpr int kVecOff = kRedOff + kRedBytes;
constexpr int kVecFloats = 2048;     // norm gain (H <= 1024) or the heads' bias tiles
constexpr int kPartOff = kVecOff + kVecFloats * 4;
constexpr int kBarOff = kPartOff + kConsumerWarps * kMaxCols * 4;
constexpr int kFlagOff = kBarOff + 2 * kNumSlots * 8;
constexpr int kRmsOff = kFlagOff + 64;
constexpr int kInfoOff = kRmsOff + kMaxCols * 4;
constexpr int kSmemBytes = kInfoOff + (int)((sizeof(CallInfo) + 15) / 16 * 16);
static_assert(kSmemBytes <= 227 * 1024, "frame kernel shared memory exceeds the per-CTA limit");

// The dynamic shared memory of the persistent kernels: functions that are not inlined
// (called once per call or per layer) rebuild the layout from it rather than taking the
// consumer state by reference, so the inlined stage code keeps its parameters in the
// constant bank.
extern __shared__ __align__(1024) uint8_t mcd_dyn_smem[];

__device__ __forceinline__ Smem smem_layout(uint8_t* base) {
  Smem s;
  s.ring = base + kRingOff;
  s.act = reinterpret_cast<float*>(base + kActOff);
  s.bfrag = base + kBfragOff;
  s.red = reinterpret_cast<float*>(base + kRedOff);
  s.vec = reinterpret_cast<float*>(base + kVecOff);
  s.part = reinterpret_cast<float*>(base + kPartOff);
  s.full = reinterpret_cast<uint64_t*>(base + kBarOff);
  s.empty = s.full + kNumSlots;
  s.flags = reinterpret_cast<int*>(base + kFlagOff);
  s.inv_rms = reinterpret_cast<float*>(base + kRmsOff);
  s.ci = reinterpret_cast<CallInfo*>(base + kInfoOff);
  return s;
}

// ------------------------------------------------------------------------------------
// Schedule shared by producer and consumers
// ------------------------------------------------------------------------------------
__device__ __forceinline__ int n_stages(const FrameParams& p) { return 4 * p.L + 1; }
__device__ __forceinline__ int stage_kind(int si, int L) { return si < 4 * L ? (si & 3) : MAT_HEAD; }

__device__ __forceinline__ int stage_units(const FrameParams& p, int si, int n_heads) {
  const int kind = stage_kind(si, p.L);
  return kind == MAT_HEAD ? n_heads * p.g[MAT_HEAD].n_units : p.g[kind].n_units;
}

// `heads` lists the positions P of the LM heads the call streams (heads stage only).
__device__ __forceinline__ const uint8_t* unit_src(const FrameParams& p, int si, int u, const int* heads) {
  const int kind = stage_kind(si, p.L);
  const MatGeom& g = p.g[kind];
  if (kind == MAT_HEAD) {
    const int hi = u / g.n_units, uu = u % g.n_units;
    return p.w_head + (long long)(heads[hi] - 1) * g.stride + (long long)uu * g.unit_bytes;
  }
  const int layer = si >> 2;
  const uint8_t* base = kind == MAT_QKV ? p.w_qkv : kind == MAT_WO ? p.w_wo : kind == MAT_GU ? p.w_gu : p.w_wd;
  return base + (long long)layer * g.stride + (long long)u * g.unit_bytes;
}

// Units [first, end) step `step` of stage si for this CTA: strided with rotation for most
// backbone stages; one contiguous block for the LM heads (a CTA mostly reads one head) and
// for the down projection (a CTA's units mostly share one k-chunk, so one operand).
struct UnitRange {
  int first, end, step;
};
__device__ __forceinline__ UnitRange unit_range(int si, int L, int n, int cta, int rot, int n_cta) {
  if (stage_kind(si, L) == MAT_HEAD || stage_kind(si, L) == MAT_WD) {
    // (cta + 1) * n < 2^32 for every supported shape: 32-bit division
    const unsigned un = (unsigned)n, uc = (unsigned)n_cta;
    return UnitRange{(int)(((unsigned)cta * un) / uc), (int)(((unsigned)(cta + 1) * un) / uc), 1};
  }
  const int f = cta - rot;                // 0 <= cta, rot < n_cta
  return UnitRange{f < 0 ? f + n_cta : f, n, n_cta};
}

// ------------------------------------------------------------------------------------
// Producer side of the ring (one thread)
// ------------------------------------------------------------------------------------
// Copy `bytes` from src into ring slot issued % kNumSlots once the consumers have released
// it; false if the wait gave up (error, stop flag or timeout).
__device__ __forceinline__ bool ring_issue(const FrameParams& p, Smem& sm, uint32_t& issued, const uint8_t* src,
                                           uint32_t bytes, uint64_t pol, const volatile int* stop) {
  const uint32_t slot = issued % kNumSlots;
  if (issued >= (uint32_t)kNumSlots) {
    if (!wait_mbar(&sm.empty[slot], ((issued / kNumSlots) - 1u) & 1u, p.err, p.wait_ns, stop)) return false;
  }
  mbar_arrive_expect_tx(&sm.full[slot], bytes);
  bulk_g2s(sm.ring + (size_t)slot * kSlotBytes, src, bytes, &sm.full[slot], pol);
  ++issued;
  return true;
}

// Every issued copy must land before the CTA may exit (bounded wait per slot).
__device__ __forceinline__ void ring_drain(const FrameParams& p, Smem& sm, uint32_t issued) {
  const uint32_t first = issued > (uint32_t)kNumSlots ? issued - kNumSlots : 0u;
  for (uint32_t i = first; i < issued; ++i) {
    const uint32_t slot = i % kNumSlots;
    uint64_t t0 = globaltimer();
    while (!mbar_try_wait(&sm.full[slot], (i / kNumSlots) & 1u)) {
      if (globaltimer() - t0 > p.wait_ns) {
        atomicCAS(p.err, 0, (int)MCD_ERR_TIMEOUT);
        break;
      }
    }
  }
}

// ------------------------------------------------------------------------------------
// Consumer helpers
// ------------------------------------------------------------------------------------
struct Cons {
  const FrameParams& p;
  Smem& sm;
  uint32_t seq;   // units consumed (ring sequence)
  int rot;
  bool abort_;
  uint8_t* op;    // B operand of the current stage (in the 64 KB work region act + bfrag)
  __device__ Cons(const FrameParams& pp, Smem& s)
      : p(pp), sm(s), seq(0), rot(0), abort_(false), op(reinterpret_cast<uint8_t*>(s.act)) {}
};

// Offset of the Wo operand in the work region: past the attention scratch (< 48 KB).
constexpr int kWoOperandOff = 48 * 1024;

// Optional profiling stamps (%globaltimer, ns), 128 per call.  Slots: 0 call start;
// 1 top-k inputs ready; 2 top-k done (CTA 0); 3 top-k done (last CTA); 4..7 acceptance
// start / records staged / decided / end.  Stage s (0..4L, 4l+k = layer l step k, 4L =
// heads) at 8+4s: +0 inputs ready (CTA 0), +1 first unit's weights in smem (CTA 0),
// +2 last epilogue done and +3 signalled (latest CTA).
constexpr int kTimelineSlots = 128;
// (Indexed by verify round; noisy-target passes are not stamped.)
__device__ __forceinline__ void timeline_p(const FrameParams& p, const CallInfo* ci, int idx, bool any_cta = false) {
  if (p.timeline && threadIdx.x == 0 && (any_cta || blockIdx.x == 0) && idx < kTimelineSlots && !ci->emu &&
      ci->round0 < kMaxCalls)
    p.timeline[ci->round0 * kTimelineSlots + idx] = globaltimer();
}
__device__ __forceinline__ void timeline(const Cons& c, int, int idx, bool any_cta = false) {
  timeline_p(c.p, c.sm.ci, idx, any_cta);
}
__device__ __forceinline__ void timeline_max(const Cons& c, int, int idx) {
  const CallInfo* ci = c.sm.ci;
  if (c.p.timeline && threadIdx.x == 0 && idx < kTimelineSlots && !ci->emu && ci->round0 < kMaxCalls)
    atomicMax(c.p.timeline + ci->round0 * kTimelineSlots + idx, (unsigned long long)globaltimer());
}

__device__ __forceinline__ bool cons_wait(Cons& c, const unsigned* ctr, unsigned target) {
  if (threadIdx.x == 0) {
    bool ok = wait_counter(ctr, target, c.p.err, c.p.wait_ns);
    if (!ok) c.sm.flags[1] = 1;
  }
  consumer_sync();
  if (*(volatile int*)&c.sm.flags[1]) c.abort_ = true;
  return !c.abort_;
}

__device__ __forceinline__ void cons_signal(Cons& c, unsigned* ctr, int call, int slot) {
  consumer_sync();
  timeline_max(c, call, slot);
  if (threadIdx.x == 0) red_release_add(ctr, 1u);
  timeline_max(c, call, slot + 1);
}

// Operand geometry of a call with ncols packed columns: ncp = 2^ceil(log2 ncols) columns,
// NT = ncp / 8 n-tiles (at least 1).  Up to 16
// columns the activations are a bf16 hi + lo pair (16 B per fragment entry, about 16
// mantissa bits); beyond that a single bf16 (8 B per entry).
__device__ __forceinline__ int col_log2(int ncols) {
  return ncols <= 1 ? 0 : ncols <= 2 ? 1 : ncols <= 4 ? 2 : ncols <= 8 ? 3 : ncols <= 16 ? 4 : 5;
}
__device__ __forceinline__ int n_tiles(int ncols) { return max(1, (1 << col_log2(ncols)) >> 3); }
__device__ __forceinline__ bool hilo_operand(int ncols) { return ncols <= 16; }

// Activation operand in one pass.  `ld(n, k, VecW{})` returns elements k .. k+W-1 of column
// n (W = 2 or 4, k a multiple of W) from global or shared memory; `gain` (shared, may be
// null) multiplies them per input index; with want_ss the per-column 1/rms of the raw values
// lands in inv_rms; store_raw (may be null) receives the raw values as fp32 rows
// [ncols][ldk].  bf16 weights get B fragments of mma.m16n8k16: entry ((kt0 + kt) * NT + nt,
// lane) holds column nt*8 + lane/4, inputs kt*16 + 2(lane%4) + {0,1,8,9}; fp32 weights get
// fp32 rows [ncols][ldk] from column kt0*16.
//
// Narrow form (up to 8 columns): thread (column, lane % 4) loads its two input pairs of a
// k-tile as 8-byte pieces and writes the whole entry; ncp = 2^ceil(log2 ncols) columns are
// written (columns >= ncols as zeros).  Every load of a batch is issued before any of its
// stores (one memory round trip per 1024 entries).
template <int WT, bool WIDE, class Ld>
__device__ __forceinline__ void prep_operand_pairs(Cons& c, int ncols, int Kdim, int kt0, int ldk, const float* gain,
                                                   bool want_ss, Ld ld, float* store_raw) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int lg = col_log2(ncols), NT = WIDE ? n_tiles(ncols) : 1;
  const bool hilo = WIDE ? hilo_operand(ncols) : true;
  const int n = (tid >> 2) & ((1 << lg) - 1), t = tid & 3;
  const bool live = n < ncols;
  const int items = (Kdim >> 4) << (2 + lg);       // (k-tile, column, t)
  constexpr int kE = 4;
  float ss = 0.f;
  for (int base = 0; base < items; base += kE * kConsumerThreads) {
    float2 va[kE], vb[kE];
#pragma unroll
    for (int e = 0; e < kE; ++e) {
      const int i = base + tid + e * kConsumerThreads;
      va[e] = make_float2(0.f, 0.f);
      vb[e] = make_float2(0.f, 0.f);
      if (i < items && live) {
        const int k0 = ((i >> (2 + lg)) << 4) + 2 * t;
        va[e] = ld(n, k0, Vec2{});
        vb[e] = ld(n, k0 + 8, Vec2{});
      }
    }
#pragma unroll
    for (int e = 0; e < kE; ++e) {
      const int i = base + tid + e * kConsumerThreads;
      if (i < items) {
        const int kt = i >> (2 + lg), k0 = (kt << 4) + 2 * t;
        float2 x01 = va[e], x89 = vb[e];
        ss += x01.x * x01.x + x01.y * x01.y + x89.x * x89.x + x89.y * x89.y;
        if (store_raw && live) {
          *reinterpret_cast<float2*>(store_raw + (size_t)n * ldk + k0) = x01;
          *reinterpret_cast<float2*>(store_raw + (size_t)n * ldk + k0 + 8) = x89;
        }
        if (gain) {
          const float2 g01 = *reinterpret_cast<const float2*>(gain + k0);
          const float2 g89 = *reinterpret_cast<const float2*>(gain + k0 + 8);
          x01.x *= g01.x;
          x01.y *= g01.y;
          x89.x *= g89.x;
          x89.y *= g89.y;
        }
        if (WT != MCD_WEIGHT_F32) {
          const int entry = ((kt0 + kt) * NT + (n >> 3)) * 32 + 4 * (n & 7) + t;
          const uint32_t h01 = pack_bf16x2(x01.x, x01.y), h89 = pack_bf16x2(x89.x, x89.y);
          if (hilo) {
            const uint32_t l01 = pack_bf16x2(x01.x - bf16_lo_f32(h01), x01.y - bf16_hi_f32(h01));
            const uint32_t l89 = pack_bf16x2(x89.x - bf16_lo_f32(h89), x89.y - bf16_hi_f32(h89));
            reinterpret_cast<uint4*>(c.op)[entry] = make_uint4(h01, h89, l01, l89);
          } else {
            reinterpret_cast<uint2*>(c.op)[entry] = make_uint2(h01, h89);
          }
        } else {
          float* xs = reinterpret_cast<float*>(c.op) + n * ldk + kt0 * 16 + k0;
          *reinterpret_cast<float2*>(xs) = x01;
          *reinterpret_cast<float2*>(xs + 8) = x89;
        }
      }
    }
  }
  if (want_ss) {
    // lanes of one column: t (bits 0-1) and the k-tile bits above the column bits
#pragma unroll
    for (int off = 1; off < 32; off <<= 1)
      if (off < 4 || off >= (4 << lg)) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, off);
    if (lane < (4 << lg) && t == 0) c.sm.part[warp * kMaxCols + n] = ss;
  }
  consumer_sync();
  if (want_ss) {
    if (tid < ncols) {
      // warp w holds columns 8w .. 8w+7 (mod ncp): only those warps' partials exist
      const int ncp = 1 << lg, own = (tid & ~7) & (ncp - 1);
      float s = 0.f;
#pragma unroll
      for (int w = 0; w < kConsumerWarps; ++w)
        if (((8 * w) & (ncp - 1)) == own) s += c.sm.part[w * kMaxCols + tid];  // fixed order
      c.sm.inv_rms[tid] = rsqrtf(__fmul_rn(s, __frcp_rn((float)Kdim)) + c.p.eps);
    }
    // no barrier: inv_rms is read only by epilogues, which follow the chunk barrier of the
    // stage, and part / inv_rms are rewritten only after the stage's closing barrier
  }
}

// Wide form (up to 32 columns): only the ncols live columns are written (an mma output
// column depends only on its own B column and columns >= ncols are never read back).
// Threads work in quads: quad j serves column j % ncols and k-tiles j / ncols, + R, ...
// (R = 64 / ncols quads per column), each thread one 16-byte piece (4 inputs) of a k-tile,
// whose two input pairs it writes as half entries.  Every load of a batch of kE pieces is
// issued before any of its stores.
template <int WT, bool WIDE, class Ld>
__device__ __forceinline__ void prep_operand_quads(Cons& c, int ncols, int Kdim, int kt0, int ldk, const float* gain,
                                                   bool want_ss, Ld ld, float* store_raw) {
  constexpr int kQuads = kConsumerThreads / 4;
  const int tid = threadIdx.x, q = tid & 3, quad = tid >> 2;
  const int NT = WIDE ? n_tiles(ncols) : 1;
  const bool hilo = WIDE ? hilo_operand(ncols) : true;
  const int R = kQuads / ncols, n = quad % ncols, r = quad / ncols;
  const bool live = r < R;
  const int nkt = Kdim >> 4;
  constexpr int kE = 8;
  float ss = 0.f;
  if (live) {
    for (int kb = r; kb < nkt; kb += kE * R) {
      float4 v[kE];
#pragma unroll
      for (int e = 0; e < kE; ++e) {
        const int kt = kb + e * R;
        v[e] = kt < nkt ? ld(n, (kt << 4) + 4 * q, Vec4{}) : make_float4(0.f, 0.f, 0.f, 0.f);
      }
#pragma unroll
      for (int e = 0; e < kE; ++e) {
        const int kt = kb + e * R;
        if (kt >= nkt) break;
        const int k0 = (kt << 4) + 4 * q;
        float4 x = v[e];
        ss += (x.x * x.x + x.y * x.y) + (x.z * x.z + x.w * x.w);
        if (store_raw) *reinterpret_cast<float4*>(store_raw + (size_t)n * ldk + k0) = x;
        if (gain) {
          const float4 g = *reinterpret_cast<const float4*>(gain + k0);
          x.x *= g.x;
          x.y *= g.y;
          x.z *= g.z;
          x.w *= g.w;
        }
        if (WT != MCD_WEIGHT_F32) {
          // inputs 4q, 4q+1 -> lane t = 2(q&1), 4q+2, 4q+3 -> t + 1; half (q >> 1) of the entry
          const int entry = ((kt0 + kt) * NT + (n >> 3)) * 32 + 4 * (n & 7) + 2 * (q & 1), half = q >> 1;
          const uint32_t h0 = pack_bf16x2(x.x, x.y), h1 = pack_bf16x2(x.z, x.w);
          if (hilo) {
            uint32_t* e4 = reinterpret_cast<uint32_t*>(c.op) + 4 * entry + half;
            e4[0] = h0;
            e4[4] = h1;
            e4[2] = pack_bf16x2(x.x - bf16_lo_f32(h0), x.y - bf16_hi_f32(h0));
            e4[6] = pack_bf16x2(x.z - bf16_lo_f32(h1), x.w - bf16_hi_f32(h1));
          } else {
            uint32_t* e2 = reinterpret_cast<uint32_t*>(c.op) + 2 * entry + half;
            e2[0] = h0;
            e2[2] = h1;
          }
        } else {
          *reinterpret_cast<float4*>(reinterpret_cast<float*>(c.op) + n * ldk + kt0 * 16 + k0) = x;
        }
      }
    }
  }
  // column sums in a fixed order: the quad's four lanes, then (ncols dividing 8) the warp's
  // quads of the column and the 8 warps, else every quad of the column
  const bool per_warp = (8 % ncols) == 0;
  if (want_ss) {
    ss += __shfl_xor_sync(0xFFFFFFFFu, ss, 1);
    ss += __shfl_xor_sync(0xFFFFFFFFu, ss, 2);
    if (per_warp) {
#pragma unroll
      for (int off = 16; off >= 4; off >>= 1)
        if (off >= 4 * ncols) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, off);
      if ((tid & 31) < 4 * ncols && q == 0) c.sm.part[(tid >> 5) * 8 + quad % 8] = ss;
    } else if (q == 0) {
      c.sm.part[quad] = ss;                    // quad sums (0 for idle quads)
    }
  }
  consumer_sync();
  if (want_ss && tid < ncols) {
    float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
    if (per_warp) {
#pragma unroll
      for (int w = 0; w < kConsumerWarps; w += 4) {
        s0 += c.sm.part[w * 8 + tid];
        s1 += c.sm.part[(w + 1) * 8 + tid];
        s2 += c.sm.part[(w + 2) * 8 + tid];
        s3 += c.sm.part[(w + 3) * 8 + tid];
      }
    } else {
      for (int j = 0; j < R; j += 4) {
        s0 += c.sm.part[j * ncols + tid];
        if (j + 1 < R) s1 += c.sm.part[(j + 1) * ncols + tid];
        if (j + 2 < R) s2 += c.sm.part[(j + 2) * ncols + tid];
        if (j + 3 < R) s3 += c.sm.part[(j + 3) * ncols + tid];
      }
    }
    const float s = (s0 + s1) + (s2 + s3);
    c.sm.inv_rms[tid] = rsqrtf(__fmul_rn(s, __frcp_rn((float)Kdim)) + c.p.eps);
    // no barrier: inv_rms is read only by epilogues, which follow the chunk barrier of the
    // stage, and part / inv_rms are rewritten only after the stage's closing barrier
  }
}

template <int WT, bool WIDE, class Ld>
__device__ __forceinline__ void prep_operand(Cons& c, int ncols, int Kdim, int kt0, int ldk, const float* gain,
                                             bool want_ss, Ld ld, float* store_raw = nullptr) {
  if constexpr (WIDE)
    prep_operand_quads<WT, WIDE>(c, ncols, Kdim, kt0, ldk, gain, want_ss, ld, store_raw);
  else
    prep_operand_pairs<WT, WIDE>(c, ncols, Kdim, kt0, ldk, gain, want_ss, ld, store_raw);
}

// Warp roles in a unit: m-tile mi of Mu, n-tile group gn of Gn (ntpw n-tiles each) and
// k-group kg of Gk, with Mu * Gn * Gk = 8 warps.  bf16 weights spread the n-tiles over the
// warps (short reduction buffer); fp32 weights keep Gn = 1 so each warp's fp32 sums stay
// as short as with one n-tile (the reduction order does not depend on the column count).
struct WarpRole {
  int Gn, ntpw, lg_ntpw, Gk, kts, mi, gn, kg;
};
// (Mu, NT and the warp-group counts are powers of two and Gk divides Ku: shifts instead of
// divisions.)
__device__ __forceinline__ int ilog2(int v) { return 31 - __clz(v); }
__device__ __forceinline__ WarpRole warp_role(const MatGeom& g, int NT, int warp, bool split_n) {
  WarpRole w;
  const int lmu = ilog2(g.Mu), lnt = ilog2(NT);
  const int lgn = split_n ? min(lnt, 3 - lmu) : 0;        // kConsumerWarps = 8
  w.Gn = 1 << lgn;
  w.lg_ntpw = lnt - lgn;
  w.ntpw = 1 << w.lg_ntpw;
  const int lgk = 3 - lmu - lgn;
  w.Gk = 1 << lgk;
  w.kts = g.Ku >> lgk;
  w.mi = warp & (g.Mu - 1);
  const int rest = warp >> lmu;
  w.gn = rest & (w.Gn - 1);
  w.kg = rest >> lgn;
  return w;
}

// Multiply the unit in ring slot `slotp` with the prepared operand of k-chunk kc; the
// warp's partial tiles (its m-tile, its n-tiles, over its k-group) land in the reduction
// buffer of chunk unit r in mma C-fragment order.
template <int WT, bool WIDE>
__device__ __forceinline__ void unit_mma(Cons& c, const MatGeom& g, const WarpRole& w, int NT, bool hilo,
                                         const uint8_t* slotp, int Kdim, int kc, int r) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int Ku = g.Ku, kt0 = kc * Ku + w.kg * w.kts;
  float4* red = reinterpret_cast<float4*>(c.sm.red) + ((size_t)r * kConsumerWarps + warp) * w.ntpw * 32;
  if (WT != MCD_WEIGHT_F32) {
    // A fragment of k-tile t: 16 bytes per lane (bf16) or 8 bytes widened to bf16 (W8A16)
    const size_t a0i = (size_t)(w.mi * Ku + w.kg * w.kts) * 32 + lane;
    auto load_a = [&](int t) -> uint4 {
      if (WT == MCD_WEIGHT_BF16) return reinterpret_cast<const uint4*>(slotp)[a0i + (size_t)t * 32];
      return widen_i8x8(reinterpret_cast<const uint2*>(slotp)[a0i + (size_t)t * 32]);
    };
    const int ntpw = WIDE ? w.ntpw : 1;
    for (int ntl = 0; ntl < ntpw; ++ntl) {
      const int nt = WIDE ? w.gn * w.ntpw + ntl : 0;
      float a0[4] = {0.f, 0.f, 0.f, 0.f}, a1[4] = {0.f, 0.f, 0.f, 0.f};
      if (!WIDE || hilo) {
        const uint4* B = reinterpret_cast<const uint4*>(c.op) + ((size_t)kt0 * NT + nt) * 32 + lane;
#pragma unroll 8
        for (int t = 0; t < w.kts; ++t) {
          const uint4 a = load_a(t);
          const uint4 bb = B[(size_t)t * NT * 32];
          mma_bf16_16816(a0, a, bb.x, bb.y);
          mma_bf16_16816(a1, a, bb.z, bb.w);
        }
      } else {
        const uint2* B = reinterpret_cast<const uint2*>(c.op) + ((size_t)kt0 * NT + nt) * 32 + lane;
#pragma unroll 8
        for (int t = 0; t < w.kts; t += 2) {
          const uint4 a = load_a(t);
          const uint2 bb = B[(size_t)t * NT * 32];
          mma_bf16_16816(a0, a, bb.x, bb.y);
          if (t + 1 < w.kts) {
            const uint4 a2 = load_a(t + 1);
            const uint2 b2 = B[(size_t)(t + 1) * NT * 32];
            mma_bf16_16816(a1, a2, b2.x, b2.y);
          }
        }
      }
      red[ntl * 32 + lane] = make_float4(a0[0] + a1[0], a0[1] + a1[1], a0[2] + a1[2], a0[3] + a1[3]);
    }
  } else {
    // fp32 weights: lane = (row rr, k-half kh) holds 8 consecutive inputs of a tile row
    const int rr = lane & 15, kh = lane >> 4;
    const float* xs = reinterpret_cast<const float*>(c.op);
    const float4* A = reinterpret_cast<const float4*>(slotp) + (size_t)(w.mi * Ku + w.kg * w.kts) * 64 + lane * 2;
    const int ntpw = WIDE ? w.ntpw : 1;
    for (int ntl = 0; ntl < ntpw; ++ntl) {
      const int n0 = (WIDE ? w.gn * w.ntpw + ntl : 0) * 8;
      float acc[8];
#pragma unroll
      for (int n = 0; n < 8; ++n) acc[n] = 0.f;
      for (int t = 0; t < w.kts; ++t) {
        const float4 w0 = A[t * 64], w1 = A[t * 64 + 1];
        const int col = (kt0 + t) * 16 + kh * 8;
#pragma unroll
        for (int n = 0; n < 8; ++n) {
          const float4 x0 = *reinterpret_cast<const float4*>(xs + (n0 + n) * Kdim + col);
          const float4 x1 = *reinterpret_cast<const float4*>(xs + (n0 + n) * Kdim + col + 4);
          acc[n] += w0.x * x0.x + w0.y * x0.y + w0.z * x0.z + w0.w * x0.w + w1.x * x1.x + w1.y * x1.y +
                    w1.z * x1.z + w1.w * x1.w;
        }
      }
#pragma unroll
      for (int n = 0; n < 8; ++n) acc[n] += __shfl_xor_sync(0xFFFFFFFFu, acc[n], 16);
      if (lane < 16) {
        float* rf = reinterpret_cast<float*>(red + ntl * 32);
#pragma unroll
        for (int n = 0; n < 8; ++n) rf[((rr & 7) * 4 + (n >> 1)) * 4 + (rr >> 3) * 2 + (n & 1)] = acc[n];
      }
    }
  }
}

// Sum over the k-group warps of output (row rr of m-tile mi, column c) of chunk unit r.
__device__ __forceinline__ float red_sum(const Cons& c, const MatGeom& g, const WarpRole& w, int r, int mi, int rr,
                                         int col) {
  const int nt = col >> 3, n = col & 7, gn = nt >> w.lg_ntpw, ntl = nt & (w.ntpw - 1);
  const float* red = c.sm.red;
  const int ln = (rr & 7) * 4 + (n >> 1), idx = (rr >> 3) * 2 + (n & 1);
  float v = 0.f;
#pragma unroll
  for (int kg = 0; kg < kConsumerWarps; ++kg) {
    if (kg < w.Gk) {
      const int warp = (kg * w.Gn + gn) * g.Mu + mi;
      v += red[((((size_t)r * kConsumerWarps + warp) * w.ntpw + ntl) * 32 + ln) * 4 + idx];
    }
  }
  return v;
}

// A stage's schedule for this CTA: its units, the warp roles and chunking, and the size of
// the first chunk.  It depends only on the call's shape, so a stage plans before it waits
// for its inputs and the integer work overlaps the grid barrier.
struct StagePlan {
  UnitRange ur;
  WarpRole role;
  int si, n_units, ncols, NT, cap, lg_unit, lgn, cnt0;
  bool hilo, pairs;
};
template <int WT, bool WIDE, class Key>
__device__ __forceinline__ StagePlan plan_stage(const Cons& c, int si, int n_units, int ncols, Key opkey,
                                                bool pairs_rows = false) {
  const FrameParams& p = c.p;
  const MatGeom& g = p.g[stage_kind(si, p.L)];
  StagePlan sp;
  sp.si = si;
  sp.n_units = n_units;
  sp.ncols = ncols;
  sp.pairs = pairs_rows;
  sp.ur = unit_range(si, p.L, n_units, blockIdx.x, c.rot, p.n_cta);
  sp.NT = WIDE ? n_tiles(ncols) : 1;
  sp.hilo = WIDE ? hilo_operand(ncols) : true;
  sp.role = warp_role(g, sp.NT, threadIdx.x >> 5, WIDE && WT != MCD_WEIGHT_F32);
  // partials: kConsumerWarps * ntpw * 512 bytes per unit, kRedBytes in all
  static_assert(kRedBytes == kConsumerWarps * 512 * 4, "chunk capacity below assumes 4 single-n-tile units");
  sp.cap = max(1, min(kChunk, 4 >> sp.role.lg_ntpw));
  sp.lgn = col_log2(ncols);
  sp.lg_unit = ilog2(g.Mu) + (pairs_rows ? 3 : 4) + sp.lgn;     // outputs per unit (log2)
  sp.cnt0 = 0;
  const int u0 = sp.ur.first;
  if (u0 < sp.ur.end) {
    const int key = opkey(u0);
    int cnt = 1;
    while (cnt < sp.cap && u0 + cnt * sp.ur.step < sp.ur.end && opkey(u0 + cnt * sp.ur.step) == key) ++cnt;
    sp.cnt0 = cnt;
  }
  return sp;
}

// Run every unit of the planned stage.  Units are taken in chunks of up to kChunk
// consecutive units that share one operand (opkey(u): the k-chunk / head whose B operand
// they multiply; prep(u0, cnt, step) builds it for the chunk), as many as the reduction
// buffer holds.  Each chunk: wait for its units' weights, multiply them all, one barrier,
// then one epilogue pass epi(u, mi, rr, n, v, v8) over the live outputs (columns n < ncols;
// v8 = row rr + 8 for gate/up pairs).  QUAD: the epilogue takes rows rr0..rr0+3 of one
// column at once, epi(u, mi, rr0, n, float4 v) (not with gate/up pairs).
template <int WT, bool WIDE, bool QUAD = false, class Key, class Prep, class Epi>
__device__ __forceinline__ void run_stage(Cons& c, int call, const StagePlan& sp, int Kdim, Key opkey, Prep prep,
                                          Epi epi) {
  const FrameParams& p = c.p;
  const int si = sp.si;
  const MatGeom& g = p.g[stage_kind(si, p.L)];
  const int lane = threadIdx.x & 31;
  timeline(c, call, 8 + 4 * si);
  const UnitRange& ur = sp.ur;
  const int lgn = sp.lgn, lg_unit = sp.lg_unit, ncols = sp.ncols;
  const bool pairs_rows = sp.pairs;
  bool first_chunk = true;
  for (int u0 = ur.first; u0 < ur.end;) {
    int cnt = sp.cnt0;
    if (!first_chunk) {
      const int key = opkey(u0);
      cnt = 1;
      while (cnt < sp.cap && u0 + cnt * ur.step < ur.end && opkey(u0 + cnt * ur.step) == key) ++cnt;
    }
    prep(u0, cnt, ur.step);
#pragma unroll 1
    for (int r = 0; r < cnt; ++r) {
      const uint32_t slot = (c.seq + r) % kNumSlots;
      if (!wait_mbar(&c.sm.full[slot], ((c.seq + r) / kNumSlots) & 1u, p.err, p.wait_ns, nullptr))
        c.sm.flags[1] = 1;
      if (first_chunk && r == 0) timeline(c, call, 9 + 4 * si);
      unit_mma<WT, WIDE>(c, g, sp.role, sp.NT, sp.hilo, c.sm.ring + (size_t)slot * kSlotBytes, Kdim, 0, r);
      __syncwarp();
      if (lane == 0) mbar_arrive(&c.sm.empty[slot]);
    }
    c.seq += cnt;
    consumer_sync();
    if (*(volatile int*)&c.sm.flags[1]) {
      c.abort_ = true;
      return;
    }
    if constexpr (QUAD) {
      const int lg_q = lg_unit - 2;
      for (int o = threadIdx.x; o < (cnt << lg_q); o += kConsumerThreads) {
        const int r = o >> lg_q, q = o & ((1 << lg_q) - 1);
        const int row4 = q >> lgn, n = q & ((1 << lgn) - 1);
        if (n < ncols) {
          const int mi = row4 >> 2, rr0 = (row4 & 3) << 2;
          const float4 v = make_float4(red_sum(c, g, sp.role, r, mi, rr0, n), red_sum(c, g, sp.role, r, mi, rr0 + 1, n),
                                       red_sum(c, g, sp.role, r, mi, rr0 + 2, n),
                                       red_sum(c, g, sp.role, r, mi, rr0 + 3, n));
          epi(u0 + r * ur.step, mi, rr0, n, v);
        }
      }
    } else {
      for (int o = threadIdx.x; o < (cnt << lg_unit); o += kConsumerThreads) {
        const int r = o >> lg_unit, q = o & ((1 << lg_unit) - 1);
        const int row = q >> lgn, n = q & ((1 << lgn) - 1);
        if (n < ncols) {
          const int mi = row >> (pairs_rows ? 3 : 4), rr = row & (pairs_rows ? 7 : 15);
          const float v = red_sum(c, g, sp.role, r, mi, rr, n);
          const float v8 = pairs_rows ? red_sum(c, g, sp.role, r, mi, rr + 8, n) : 0.f;
          epi(u0 + r * ur.step, mi, rr, n, v, v8);
        }
      }
    }
    u0 += cnt * ur.step;
    first_chunk = false;
    if (u0 < ur.end) consumer_sync();
  }
  int rot = c.rot + sp.n_units;
  while (rot >= p.n_cta) rot -= p.n_cta;
  c.rot = rot;
}

// Plan and run in one step (stages whose plan cannot precede a wait).
template <int WT, bool WIDE, class Key, class Prep, class Epi>
__device__ __forceinline__ void run_stage(Cons& c, int call, int si, int n_units, int Kdim, int ncols, Key opkey,
                                          Prep prep, Epi epi, bool pairs_rows = false) {
  const StagePlan sp = plan_stage<WT, WIDE>(c, si, n_units, ncols, opkey, pairs_rows);
  run_stage<WT, WIDE>(c, call, sp, Kdim, opkey, prep, epi);
}

// Read-only vector (weights) into shared memory; no barrier (a later barrier orders it).
__device__ __forceinline__ void g2s_vec(float* dst, const float* src, int n) {
  const int n4 = n >> 2;
  for (int i = threadIdx.x; i < n4; i += kConsumerThreads)
    reinterpret_cast<float4*>(dst)[i] = __ldg(reinterpret_cast<const float4*>(src) + i);
}

template <int W> __device__ __forceinline__ vecf<W> ld_global_v(const float* q) {
  return __ldcg(reinterpret_cast<const vecf<W>*>(q));
}
template <int W> __device__ __forceinline__ vecf<W> ld_shared_v(const float* q) {
  return *reinterpret_cast<const vecf<W>*>(q);
}
// elements k .. k+W-1 of a read-only row of fp32 or bf16 values (k a multiple of W)
template <int W> __device__ __forceinline__ vecf<W> ldg_f32_v(const uint8_t* row, int k) {
  return __ldg(reinterpret_cast<const vecf<W>*>(row) + k / W);
}
template <int W> __device__ __forceinline__ vecf<W> ldg_bf16_v(const uint8_t* row, int k) {
  if constexpr (W == 4) {
    const uint2 w = __ldg(reinterpret_cast<const uint2*>(row) + (k >> 2));
    return make_float4(bf16_bits_to_f32(w.x & 0xFFFFu), bf16_bits_to_f32(w.x >> 16), bf16_bits_to_f32(w.y & 0xFFFFu),
                       bf16_bits_to_f32(w.y >> 16));
  } else {
    const uint32_t w = __ldg(reinterpret_cast<const uint32_t*>(row) + (k >> 1));
    return make_float2(bf16_bits_to_f32(w & 0xFFFFu), bf16_bits_to_f32(w >> 16));
  }
}
template <int W> __device__ __forceinline__ void add_v(vecf<W>& a, const vecf<W>& b) {
  a.x += b.x;
  a.y += b.y;
  if constexpr (W == 4) {
    a.z += b.z;
    a.w += b.w;
  }
}

}  // namespace mcd
