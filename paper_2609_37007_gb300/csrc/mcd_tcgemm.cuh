// Tensor-core GEMM on the 5th-generation tensor cores (tcgen05, TMEM accumulators) for the
// products of the batched path that are real GEMMs: D[m][n] = sum_k A[m][k] B[n][k] with A
// the weights (bf16, M x K) and B the packed activation rows (bf16, N x K), fp32 accumulation.
//
// Operands live in HBM in the "SW128 tile" layout: for every 64-wide k-slice kt, rows in
// groups of 8 form 1024-byte atoms, row r of an atom is 128 bytes (64 bf16) and its 16-byte
// chunk c sits at chunk position c ^ (r % 8).  A tile of TR rows (TR % 8 == 0) of one k-slice
// is then TR * 128 contiguous bytes that one cp.async.bulk copies into shared memory, where it
// is exactly the canonical K-major layout with 128-byte swizzle that tcgen05.mma reads
// (8-row groups 1024 bytes apart).  No tensor map is needed.
//
// gemm_tile: one CTA computes a 128 x BN tile of D (UMMA M = 128, N = BN, K = 16 per
// instruction): a producer thread streams the k-slices of A and B through a ring of as many
// stages as fit in 200 KB (4 to 6; mbarrier complete_tx), one thread issues the MMAs and
// returns each stage with tcgen05.commit, and after the last commit the four warps read the
// accumulator back from TMEM (warp w owns lanes 32w..32w+31 = rows m of the tile) and hand
// every value to the epilogue functor.  gemm_persistent (below) runs the same pipeline over
// many tiles per CTA with two TMEM accumulators, so one tile's epilogue overlaps the next
// tile's MMAs.  Every wait is bounded (wait_ns); on a timeout the CTA records
// MCD_ERR_TIMEOUT, lets the copies and MMAs it started finish, frees its TMEM and returns.
#pragma once
#include "mcd_internal.cuh"

namespace mcd {
namespace tc {

constexpr int kBM = 128;         // rows of A per tile (UMMA M)
constexpr int kBK = 64;          // k per stage: one 128-byte swizzled row
constexpr int kStageBudget = 200 * 1024;   // shared memory for the ring (stages of one k-slice)
constexpr int kThreads = 128;

// Byte offset of (row, 16-byte chunk c) of k-slice kt in the SW128 tile layout of a matrix
// with R rows.
__host__ __device__ __forceinline__ size_t sw128_offset(int R, int row, int kt, int c) {
  return (size_t)kt * R * 128 + (size_t)(row >> 3) * 1024 + (size_t)(row & 7) * 128 + (size_t)((c ^ (row & 7)) << 4);
}

// kDualA: a second A matrix (same shape) multiplies the same B into a second accumulator
// (gate and up projections side by side); kDualB: a second B operand (the low bf16 half of
// a hi + lo split) accumulates into the same accumulator.
// TMEM allocations are powers of two of at least 32 columns.
__host__ __device__ constexpr int tmem_cols_for(int cols) {
  int c = 32;
  while (c < cols) c <<= 1;
  return c;
}

template <int BN, bool kDualA = false, bool kDualB = false>
struct Layout {
  static_assert(BN % 16 == 0 && BN >= 32 && BN <= 256, "UMMA N");
  static constexpr int kABytes = kBM * 128;
  static constexpr int kBBytes = BN * 128;
  static constexpr int kStageBytes = (kDualA ? 2 : 1) * kABytes + (kDualB ? 2 : 1) * kBBytes;
  static constexpr int kTmemCols = tmem_cols_for((kDualA ? 2 : 1) * BN);
  static constexpr int kStages = kStageBudget / kStageBytes > 8 ? 8 : kStageBudget / kStageBytes;
  static constexpr int kBarOff = kStages * kStageBytes;                 // full[s], empty[s], accum
  static constexpr int kTmemSlotOff = kBarOff + (2 * kStages + 1) * 8;
  static constexpr int kFlagOff = kTmemSlotOff + 4;
  static constexpr int kSmemBytes = kFlagOff + 4 + 1024;               // + alignment slack
  static_assert(kSmemBytes <= 227 * 1024, "tensor-core GEMM stages exceed shared memory");
  static_assert(kTmemCols <= 512, "TMEM columns");
};

// Shared-memory matrix descriptor: K-major, 128-byte swizzle, 8-row groups 1024 B apart.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t smem_addr) {
  uint64_t d = 0;
  d |= (uint64_t)((smem_addr >> 4) & 0x3FFFu);            // start address
  d |= (uint64_t)1u << 16;                                 // leading byte offset (unused here)
  d |= (uint64_t)(1024u >> 4) << 32;                       // stride byte offset
  d |= (uint64_t)1u << 46;                                 // descriptor version
  d |= (uint64_t)2u << 61;                                 // 128-byte swizzle
  return d;
}

// Instruction descriptor of kind::f16: bf16 A and B (K-major), fp32 D, M = 128, N = n.
__host__ __device__ constexpr uint32_t idesc_bf16_n(int n) {
  return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(kBM >> 4) << 24);
}
template <int BN>
__host__ __device__ constexpr uint32_t idesc_bf16() {
  return idesc_bf16_n(BN);
}

__device__ __forceinline__ void umma_bf16(uint32_t tmem_d, uint64_t a, uint64_t b, uint32_t idesc, bool accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.u32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(tmem_d),
      "l"(a), "l"(b), "r"(idesc), "r"((uint32_t)accumulate)
      : "memory");
}
__device__ __forceinline__ void umma_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }

// 32 lanes x 16 consecutive fp32 columns of TMEM (lane = this thread's lane of the warp's
// quarter) into v[0..15].
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// The same load without its wait: r is defined only after tmem_wait16(r), which names the
// registers so that no use of them can move above the wait.
__device__ __forceinline__ void tmem_ld16_async(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}
__device__ __forceinline__ void tmem_wait16(uint32_t (&r)[16]) {
  asm volatile("tcgen05.wait::ld.sync.aligned;"
               : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                 "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15])
               :
               : "memory");
}

__device__ __forceinline__ uint64_t policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// Bounded wait on an mbarrier phase; false (and the error recorded) on a timeout.
__device__ __forceinline__ bool tc_wait(uint64_t* bar, uint32_t parity, int* err, unsigned long long wait_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  while (!mbar_try_wait(bar, parity)) {
    if (globaltimer() - t0 > wait_ns) {
      atomicCAS(err, 0, (int)MCD_ERR_TIMEOUT);
      return false;
    }
  }
  return true;
}

struct GemmArgs {
  const uint8_t* a;      // A in SW128 tiles, M rows
  const uint8_t* a2;     // kDualA: the second A (same layout)
  const uint8_t* b;      // B in SW128 tiles, N rows
  const uint8_t* b2;     // kDualB: the second B (same layout)
  int M, N, K;           // M % 128 == 0, N % BN == 0, K % 64 == 0
  const int* n_active;   // optional (device): columns n >= *n_active are not computed
  int* err;
  unsigned long long wait_ns;
  int bn;                // gemm_tile: 0 = tiles of BN columns; else tile x covers columns
                         // x * bn .. min(N, (x + 1) * bn) - 1 (bn a multiple of 16, <= BN)
};

// Tile pitch over N that fills n_sm SMs with one tile per CTA: T = n_sm / (M / 128) tiles
// across N (at least ceil(N / 256)), each a multiple of 16 columns.
inline int tile_pitch(int M, int N, int n_sm) {
  const int n_mt = M / kBM, units = N / 16;
  int T = n_sm / (n_mt > 1 ? n_mt : 1);
  if (T < 1) T = 1;
  if (T < (N + 255) / 256) T = (N + 255) / 256;
  if (T > units) T = units;
  return (units + T - 1) / T * 16;
}

// The tile of a CTA once its k-loop has run (gemm_tile_run).
struct TileRun {
  uint8_t* smem;   // the operand ring: idle once every MMA has completed
  uint32_t tmem;   // the accumulator(s)
  int m0, n0, nw;  // first row of A, first column and columns of the tile
  bool ok;         // every MMA completed (false after a timeout)
};

// Set-up, operand stream and MMAs of the tile of this CTA: columns n0 .. n0 + nw - 1 (by
// default x * pitch .. for x = blockIdx.x; else as given, n0 and nw multiples of 16, nw <= BN).
// false: the tile is empty (its first column at or past *n_active, or no k-slices in its
// split) and nothing is held; else every thread returns after the accumulator is complete
// (t.ok) or the tile gave up, and the CTA must call gemm_tile_free.
template <int BN, bool kDualA, bool kDualB>
__device__ __forceinline__ bool gemm_tile_run(const GemmArgs& g, TileRun& t, int n0 = -1, int nw = 0) {
  using L = Layout<BN, kDualA, kDualB>;
  extern __shared__ uint8_t tc_smem_raw[];
  const int m0 = blockIdx.y * kBM;
  if (n0 < 0) {
    const int pitch = g.bn ? g.bn : BN;
    n0 = blockIdx.x * pitch;
    nw = min(pitch, g.N - n0);                                    // this tile's columns
  }
  if (g.n_active && n0 >= __ldg(g.n_active)) return false;    // uniform over the CTA
  const int nk_all = g.K / kBK, per = (nk_all + gridDim.z - 1) / gridDim.z;
  const int kt0 = blockIdx.z * per, kt1 = min(nk_all, kt0 + per), nk = kt1 - kt0;
  if (nk <= 0) return false;
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(tc_smem_raw) + 1023) & ~(uintptr_t)1023);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L::kBarOff);
  uint64_t* empty = full + L::kStages;
  uint64_t* accum = empty + L::kStages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::kTmemSlotOff);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::kFlagOff);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < L::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accum, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"((uint32_t)L::kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0 && lane == 0) {
    // producer: k-slice kt of the A tile(s) (rows m0..) and the B tile(s) (rows n0..)
    const uint64_t pol_a = policy_evict_first(), pol_b = policy_evict_last();
    int issued = 0;
    for (int i = 0; i < nk; ++i) {
      const int s = i % L::kStages, kt = kt0 + i;
      if (i >= L::kStages && !tc_wait(&empty[s], ((i / L::kStages) - 1) & 1, g.err, g.wait_ns)) {
        *abort_flag = 1;
        break;
      }
      if (*abort_flag) break;
      uint8_t* st = smem + s * L::kStageBytes;
      const size_t ao = (size_t)kt * g.M * 128 + (size_t)m0 * 128, bo = (size_t)kt * g.N * 128 + (size_t)n0 * 128;
      const uint32_t b_bytes = (uint32_t)nw * 128u;
      mbar_arrive_expect_tx(&full[s], (kDualA ? 2 : 1) * L::kABytes + (kDualB ? 2 : 1) * b_bytes);
      bulk_g2s(st, g.a + ao, L::kABytes, &full[s], pol_a);
      if (kDualA) bulk_g2s(st + L::kABytes, g.a2 + ao, L::kABytes, &full[s], pol_a);
      uint8_t* sb = st + (kDualA ? 2 : 1) * L::kABytes;
      bulk_g2s(sb, g.b + bo, b_bytes, &full[s], pol_b);
      if (kDualB) bulk_g2s(sb + L::kBBytes, g.b2 + bo, b_bytes, &full[s], pol_b);
      ++issued;
    }
    // every issued copy lands before the CTA may exit
    for (int i = (issued > L::kStages ? issued - L::kStages : 0); i < issued; ++i)
      tc_wait(&full[i % L::kStages], (i / L::kStages) & 1, g.err, g.wait_ns);
  } else if (warp == 1 && lane == 0) {
    // MMA issuer
    const uint32_t idesc = idesc_bf16_n(nw);
    for (int i = 0; i < nk; ++i) {
      const int s = i % L::kStages;
      if (!tc_wait(&full[s], (i / L::kStages) & 1, g.err, g.wait_ns)) {
        *abort_flag = 1;
        break;
      }
      if (*abort_flag) break;
      tc_fence_after();
      const uint32_t sa = smem_u32(smem + s * L::kStageBytes);
      const uint32_t sb = sa + (kDualA ? 2 : 1) * L::kABytes;
#pragma unroll
      for (int j = 0; j < kBK / 16; ++j) {
        const bool acc = (i | j) != 0;
        umma_bf16(tmem, sw128_desc(sa + 32 * j), sw128_desc(sb + 32 * j), idesc, acc);
        if (kDualB) umma_bf16(tmem, sw128_desc(sa + 32 * j), sw128_desc(sb + L::kBBytes + 32 * j), idesc, true);
        if (kDualA)
          umma_bf16(tmem + BN, sw128_desc(sa + L::kABytes + 32 * j), sw128_desc(sb + 32 * j), idesc, acc);
      }
      umma_commit(&empty[s]);         // the stage is free once these MMAs have read it
    }
    umma_commit(accum);               // every MMA issued so far has completed
  }
  t.ok = tc_wait(accum, 0, g.err, g.wait_ns) && !*abort_flag;
  __syncwarp();                       // the .sync.aligned TMEM loads need whole warps
  tc_fence_after();
  t.smem = smem;
  t.tmem = tmem;
  t.m0 = m0;
  t.n0 = n0;
  t.nw = nw;
  return true;
}

// Every thread of the CTA, after the last TMEM load: the accumulator's columns are freed.
template <int BN, bool kDualA, bool kDualB>
__device__ __forceinline__ void gemm_tile_free(const TileRun& t) {
  using L = Layout<BN, kDualA, kDualB>;
  tc_fence_before();
  __syncthreads();
  if ((threadIdx.x >> 5) == 1)
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(t.tmem), "r"((uint32_t)L::kTmemCols)
                 : "memory");
}

// The GEMM body for the tile of rows m0 = blockIdx.y * 128 of A and n0 = blockIdx.x * BN of B
// over the k-slices of split blockIdx.z of gridDim.z (the CTAs that share an A tile are
// adjacent in launch order, so the weights stream from HBM about once while the activation
// tiles stay in L2); epi(m, n, v, v2) for every m and n of the tile (each thread: one m, BN
// values of n in order; v2 = the second accumulator with kDualA, else 0).  A tile whose
// first column is at or past *n_active returns at once.  n0 >= 0: the tile's columns are
// n0 .. n0 + nw - 1 instead (see gemm_tile_run).
template <int BN, bool kDualA, bool kDualB, class Epi>
__device__ __forceinline__ void gemm_tile(const GemmArgs& g, Epi epi, int n0 = -1, int nw = 0) {
  TileRun t;
  if (!gemm_tile_run<BN, kDualA, kDualB>(g, t, n0, nw)) return;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m0 = t.m0;
  n0 = t.n0;
  nw = t.nw;
  const uint32_t tmem = t.tmem;
  // epilogue: every warp, after the accumulator is complete
  if (t.ok) {
    // warp w reads TMEM lanes 32 (w % 4) ..; with more than four warps the 16-column chunks
    // are shared out (chunk c to the warps w / 4 == c mod (warps / 4))
    const int quarter = warp & 3, part = warp >> 2, n_parts = (int)(blockDim.x >> 7);
    const int m = m0 + quarter * 32 + lane, n_ch = nw >> 4;
    const uint32_t lane_base = tmem + ((uint32_t)(quarter * 32) << 16);
    if (kDualA) {
#pragma unroll 1
      for (int ch = part; ch < n_ch; ch += n_parts) {
        float v[16], v2[16];
        tmem_ld16(lane_base + (uint32_t)(16 * ch), v);
        tmem_ld16(lane_base + (uint32_t)(BN + 16 * ch), v2);
#pragma unroll
        for (int j = 0; j < 16; ++j) epi(m, n0 + 16 * ch + j, v[j], v2[j]);
      }
    } else if (part < n_ch) {
      // the next chunk's TMEM load is in flight while this chunk's values are stored (two
      // register sets, alternating)
      uint32_t ra[16], rb[16];
      auto store = [&](const uint32_t (&r)[16], int ch) {
#pragma unroll
        for (int j = 0; j < 16; ++j) epi(m, n0 + 16 * ch + j, __uint_as_float(r[j]), 0.f);
      };
      int ch = part;
      tmem_ld16_async(lane_base + (uint32_t)(16 * ch), ra);
      tmem_wait16(ra);
#pragma unroll 1
      while (true) {
        int nx = ch + n_parts;
        if (nx < n_ch) tmem_ld16_async(lane_base + (uint32_t)(16 * nx), rb);
        store(ra, ch);
        if (nx >= n_ch) break;
        tmem_wait16(rb);
        ch = nx;
        nx = ch + n_parts;
        if (nx < n_ch) tmem_ld16_async(lane_base + (uint32_t)(16 * nx), ra);
        store(rb, ch);
        if (nx >= n_ch) break;
        tmem_wait16(ra);
        ch = nx;
      }
    }
  }
  gemm_tile_free<BN, kDualA, kDualB>(t);
}

// ---- persistent form ----------------------------------------------------------------------
// Tiles t = blockIdx.x, blockIdx.x + gridDim.x, ... over (n tile fastest, then m tile, then
// k split) of an (N / BN) x (M / 128) x splits grid.  Six warps: warp 0 streams k-slices
// through the shared-memory ring across tile boundaries, warp 1 issues the MMAs into one of
// two TMEM accumulator buffers (tile i uses buffer i % 2), warps 2..5 read a finished buffer
// back (warp w: TMEM lanes 32 (w % 4) ..) while the MMAs of the next tile already run, then
// release it.  epi(m, n, split, v, v2).  Tiles whose first column is at or past *n_active are
// skipped by every role alike.
constexpr int kPThreads = 192;
template <int BN, bool kDualA, bool kDualB>
struct PLayout {
  using L = Layout<BN, kDualA, kDualB>;
  static constexpr int kAccCols = (kDualA ? 2 : 1) * BN;     // one accumulator buffer
  static constexpr int kTmemCols = tmem_cols_for(2 * kAccCols);
  static_assert(kTmemCols <= 512, "TMEM columns");
  static constexpr int kBarOff = L::kStages * L::kStageBytes;  // full[S], empty[S], acc_full[2], acc_empty[2], drain
  static constexpr int kTmemSlotOff = kBarOff + (2 * L::kStages + 5) * 8;
  static constexpr int kFlagOff = kTmemSlotOff + 4;
  static constexpr int kSmemBytes = kFlagOff + 4 + 1024;
  static_assert(kSmemBytes <= 227 * 1024, "tensor-core GEMM stages exceed shared memory");
};

template <int BN, bool kDualA, bool kDualB, class Epi>
__device__ __forceinline__ void gemm_persistent(const GemmArgs& g, int splits, Epi epi) {
  using L = Layout<BN, kDualA, kDualB>;
  using PL = PLayout<BN, kDualA, kDualB>;
  constexpr int S = L::kStages;
  extern __shared__ uint8_t tc_smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(tc_smem_raw) + 1023) & ~(uintptr_t)1023);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + PL::kBarOff);
  uint64_t* empty = full + S;
  uint64_t* acc_full = empty + S;
  uint64_t* acc_empty = acc_full + 2;
  uint64_t* drain = acc_empty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + PL::kTmemSlotOff);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + PL::kFlagOff);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_nt = g.N / BN, n_mt = g.M / kBM, n_tiles = n_nt * n_mt * splits;
  const int nk_all = g.K / kBK, per = (nk_all + splits - 1) / splits;
  const int n_live = g.n_active ? *g.n_active : g.N;
  // tile t -> (n0, m0, split, k-slice range); false for a skipped tile
  auto tile_of = [&](int t, int& n0, int& m0, int& z, int& kt0, int& nk) {
    const int nt = t % n_nt, rest = t / n_nt;
    n0 = nt * BN;
    m0 = (rest % n_mt) * kBM;
    z = rest / n_mt;
    kt0 = z * per;
    nk = min(nk_all, kt0 + per) - kt0;
    return n0 < n_live && nk > 0;
  };

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], 4);            // the four epilogue warps
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"((uint32_t)PL::kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {                          // producer
      const uint64_t pol_a = policy_evict_first(), pol_b = policy_evict_last();
      uint32_t c = 0;                         // k-slices issued
      for (int t = blockIdx.x; t < n_tiles && !*abort_flag; t += gridDim.x) {
        int n0, m0, z, kt0, nk;
        if (!tile_of(t, n0, m0, z, kt0, nk)) continue;
        for (int i = 0; i < nk; ++i, ++c) {
          const int s = c % S;
          if (c >= (uint32_t)S && !tc_wait(&empty[s], ((c / S) - 1) & 1, g.err, g.wait_ns)) {
            *abort_flag = 1;
            break;
          }
          if (*abort_flag) break;
          const int kt = kt0 + i;
          uint8_t* st = smem + s * L::kStageBytes;
          const size_t ao = (size_t)kt * g.M * 128 + (size_t)m0 * 128, bo = (size_t)kt * g.N * 128 + (size_t)n0 * 128;
          mbar_arrive_expect_tx(&full[s], L::kStageBytes);
          bulk_g2s(st, g.a + ao, L::kABytes, &full[s], pol_a);
          if (kDualA) bulk_g2s(st + L::kABytes, g.a2 + ao, L::kABytes, &full[s], pol_a);
          uint8_t* sb = st + (kDualA ? 2 : 1) * L::kABytes;
          bulk_g2s(sb, g.b + bo, L::kBBytes, &full[s], pol_b);
          if (kDualB) bulk_g2s(sb + L::kBBytes, g.b2 + bo, L::kBBytes, &full[s], pol_b);
        }
      }
      // every issued copy lands before the CTA may exit
      for (uint32_t i = c > (uint32_t)S ? c - S : 0u; i < c; ++i) tc_wait(&full[i % S], (i / S) & 1, g.err, g.wait_ns);
    }
  } else if (warp == 1) {
    if (lane == 0) {                          // MMA issuer
      constexpr uint32_t idesc = idesc_bf16<BN>();
      uint32_t c = 0;                         // k-slices consumed
      int i_tile = 0;                         // tiles computed by this CTA
      for (int t = blockIdx.x; t < n_tiles && !*abort_flag; t += gridDim.x) {
        int n0, m0, z, kt0, nk;
        if (!tile_of(t, n0, m0, z, kt0, nk)) continue;
        const int b = i_tile & 1, v = i_tile >> 1;
        if (v >= 1 && !tc_wait(&acc_empty[b], (v - 1) & 1, g.err, g.wait_ns)) {
          *abort_flag = 1;
          break;
        }
        tc_fence_after();
        const uint32_t acc = tmem + (uint32_t)(b * PL::kAccCols);
        for (int i = 0; i < nk; ++i, ++c) {
          const int s = c % S;
          if (!tc_wait(&full[s], (c / S) & 1, g.err, g.wait_ns)) {
            *abort_flag = 1;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + s * L::kStageBytes);
          const uint32_t sb = sa + (kDualA ? 2 : 1) * L::kABytes;
#pragma unroll
          for (int j = 0; j < kBK / 16; ++j) {
            const bool ac = (i | j) != 0;
            umma_bf16(acc, sw128_desc(sa + 32 * j), sw128_desc(sb + 32 * j), idesc, ac);
            if (kDualB) umma_bf16(acc, sw128_desc(sa + 32 * j), sw128_desc(sb + L::kBBytes + 32 * j), idesc, true);
            if (kDualA)
              umma_bf16(acc + BN, sw128_desc(sa + L::kABytes + 32 * j), sw128_desc(sb + 32 * j), idesc, ac);
          }
          umma_commit(&empty[s]);
        }
        umma_commit(&acc_full[b]);            // the tile's accumulator is complete
        ++i_tile;
      }
    }
  } else {
    // epilogue warps 2..5: TMEM lane quarter (warp % 4)
    const int q = warp & 3;
    int i_tile = 0;
    for (int t = blockIdx.x; t < n_tiles; t += gridDim.x) {
      int n0, m0, z, kt0, nk;
      if (!tile_of(t, n0, m0, z, kt0, nk)) continue;
      const int b = i_tile & 1, v = i_tile >> 1;
      const bool ok = tc_wait(&acc_full[b], v & 1, g.err, g.wait_ns) && !*abort_flag;
      __syncwarp();
      tc_fence_after();
      if (!ok) {
        *abort_flag = 1;
        break;
      }
      const int m = m0 + q * 32 + lane;
      const uint32_t base = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * PL::kAccCols);
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 16) {
        float vv[16], v2[16];
        tmem_ld16(base + (uint32_t)c0, vv);
        if (kDualA) tmem_ld16(base + (uint32_t)(BN + c0), v2);
#pragma unroll
        for (int j = 0; j < 16; ++j) epi(m, n0 + c0 + j, z, vv[j], kDualA ? v2[j] : 0.f);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[b]);
      ++i_tile;
    }
  }
  // every MMA this CTA issued has completed before its TMEM is freed (also after an abort)
  if (warp == 1 && lane == 0) {
    umma_commit(drain);
    tc_wait(drain, 0, g.err, g.wait_ns);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"((uint32_t)PL::kTmemCols)
                 : "memory");
  }
}

}  // namespace tc
}  // namespace mcd
