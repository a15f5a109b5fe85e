// tcgen05 GEMM for the bf16 block projections: C[M, N] = A[M, K] B[N, K]^T with
// the block's epilogues fused (bias; bias + GELU; bias + fp32 residual add; bias
// + residual + the delta scatter of Eq. 9 for the last sparse block).
//
// Persistent and warp-specialised, 320 threads per CTA.  Tiles 128 or 256
// columns wide run on CTA pairs (clusters of two, tcgen05.mma.cta_group::2):
// the pair shares a 256-row tile, each CTA holding 128 rows of A and half of
// the tile's B rows; 64-column tiles run on single CTAs (M = 128).
//   warp 0      TMA producer: A and B tiles (64 columns of K, 128-byte swizzle)
//               into a ring of shared-memory stages; a pair's loads complete on
//               the even CTA's stage barrier;
//   warp 1      owns the tensor memory; of a pair only the even CTA issues the
//               MMAs (K = 16 each), into one of two TMEM accumulators;
//   warps 2..9  epilogue: tcgen05.ld of the finished accumulator (one row per
//               thread; two warps per TMEM lane quarter, each taking half of
//               the tile's columns) while the other accumulator takes the next
//               tile's MMAs.  bf16 outputs leave through TMA stores of
//               swizzled shared-memory tiles; the fp32 residual is updated by
//               TMA reduce (bias + accumulator added into the stream in L2);
//               the scatter and 64-column tiles use a per-warp shared-memory
//               transpose and coalesced row stores (the scatter's rows are
//               prefetched into L2 during the mainloop and loaded one step
//               ahead).
// Rows beyond M are zero-filled by TMA and never stored.  Requires K % 64 == 0
// and N % BN == 0 (checked by the launcher).
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"
#include "tc_ptx.cuh"

namespace sr {
namespace {

using namespace tc;

constexpr int BM = 128, BK = 64;
constexpr int kThreads = 320;
constexpr int kEpiThreads = 256;

template <int BN, Epi E, bool kPair = false>
struct GemmCfg {
  // kPair: two CTAs of a cluster share a 256-row tile (tcgen05.mma.cta_group::2);
  // each loads its own 128 rows of A and half of the tile's B rows
  static constexpr int kRowsTile = kPair ? 2 * BM : BM;
  static constexpr int kBRows = kPair ? BN / 2 : BN;
  // the residual epilogue of pair tiles stages two 32 x 32 fp32 chunks per
  // epilogue warp in shared memory (64 KB), paid for with a shorter operand ring
  // on 256-column tiles: bias + accumulator, added into the stream by TMA
  // reduce; or, when the updated rows' norms are wanted, the residual itself,
  // loaded by TMA, updated in place and stored back
  static constexpr bool kTmaRes = E == Epi::BiasResidual && kPair;
  // bf16 outputs of tiles at least 128 columns wide leave through TMA stores
  // from a 128-byte-swizzled 32 x 64 tile per epilogue warp (4 KB)
  static constexpr bool kTmaOut = (E == Epi::Bias || E == Epi::BiasGelu) && BN >= 128;
  static constexpr int kOutTileBytes = 32 * 128;
  static constexpr int kStages = kPair ? (kTmaRes && BN == 256 ? 5 : 6) : (BN == 256 ? 4 : 6);
  static constexpr int kABytes = BM * BK * 2;        // 16 KB
  static constexpr int kBBytes = kBRows * BK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr int kTmemCols = 2 * BN;           // two accumulators
  // per epilogue warp: a 32 x 32 fp32 chunk, pitch 33 (conflict-free both ways)
  static constexpr int kStageFloats = 32 * 33;
  static constexpr int kResTileBytes = 32 * 32 * 4;  // one residual chunk (TMA box)
  static constexpr size_t kStagingBytes = kTmaRes
      ? size_t(kEpiThreads / 32) * 2 * kResTileBytes
      : kTmaOut ? size_t(kEpiThreads / 32) * kOutTileBytes
                : size_t(kEpiThreads / 32) * kStageFloats * 4;
  static constexpr size_t kSmem =
      size_t(kStages) * kStageBytes + kStagingBytes + 1024 /*align*/ + 512 /*barriers*/;
  // delta scatter on a unit's last tile: each epilogue warp stages 32-column
  // quarters of its routed rows h and of the stream rows x0 (4 KB each) in the
  // then idle operand ring, up to three quarters in flight
  static constexpr int kScatterQuarters = BN / 64;                  // per warp
  static constexpr int kScatterSlots = kScatterQuarters < 3 ? kScatterQuarters : 3;
  static constexpr int kScatterSlotBytes = 2 * 32 * 32 * 4;
  static_assert(E != Epi::BiasResidualScatter ||
                    size_t(kEpiThreads / 32) * kScatterSlots * kScatterSlotBytes <=
                        size_t(kStages) * kStageBytes,
                "scatter staging exceeds the operand ring");
};

struct Smem {
  uint64_t full[8], empty[8], tfull[2], tempty[2], drain;
  uint64_t res_full[kEpiThreads / 32][2];   // residual tiles landed (per epilogue warp)
  uint32_t tmem_base;
  int abort;
};
static_assert(sizeof(Smem) <= 512, "the barrier block must fit its reserve in GemmCfg::kSmem");
static_assert(GemmCfg<256, Epi::BiasResidual, true>::kSmem <= 232448, "pair config exceeds shared memory");
static_assert(GemmCfg<256, Epi::Bias, true>::kSmem <= 232448, "pair config exceeds shared memory");

// GELU(z) = z * Phi(z) with Phi from the erfc approximation of Abramowitz &
// Stegun, Handbook of Mathematical Functions, formula 7.1.26 (absolute error
// <= 1.5e-7): erfc(x) = t (a1 + t (a2 + t (a3 + t (a4 + t a5)))) exp(-x^2),
// t = 1 / (1 + p x), x = |z| / sqrt(2) >= 0.  Its error is far below the bf16
// rounding of the stored output.  Two values at once, with the packed fp32
// instructions.
__device__ __forceinline__ void gelu2_as7126(float& z0, float& z1) {
  const uint64_t x = mul2(pk2(fabsf(z0), fabsf(z1)),
                          pk2(0.70710678118654752f, 0.70710678118654752f));
  float d0, d1;
  up2(fma2(x, pk2(0.3275911f, 0.3275911f), pk2(1.0f, 1.0f)), d0, d1);
  const uint64_t t = pk2(rcp_approx(d0), rcp_approx(d1));
  uint64_t poly = fma2(t, pk2(1.061405429f, 1.061405429f), pk2(-1.453152027f, -1.453152027f));
  poly = fma2(t, poly, pk2(1.421413741f, 1.421413741f));
  poly = fma2(t, poly, pk2(-0.284496736f, -0.284496736f));
  poly = fma2(t, poly, pk2(0.254829592f, 0.254829592f));
  float a0, a1;
  up2(mul2(mul2(x, x), pk2(-1.4426950408889634f, -1.4426950408889634f)), a0, a1);
  // 0.5 erfc(|z| / sqrt 2) = Phi(-|z|)
  float h0, h1;
  up2(mul2(mul2(mul2(t, poly), pk2(ex2(a0), ex2(a1))), pk2(0.5f, 0.5f)), h0, h1);
  const uint64_t phi = pk2(z0 >= 0.f ? 1.0f - h0 : h0, z1 >= 0.f ? 1.0f - h1 : h1);
  up2(mul2(pk2(z0, z1), phi), z0, z1);
}

__device__ __forceinline__ void prefetch_l2(const void* p) {
  asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

// 16-byte copy from global to shared memory through L2 only (cp.async.cg);
// each thread's copies complete in commit groups it waits for
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(smem)), "l"(gmem)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
  asm volatile("cp.async.commit_group;" ::: "memory");
}
// waits until at most n of this thread's commit groups are still in flight (n < 3)
__device__ __forceinline__ void cp_async_wait_upto(int n) {
  if (n <= 0) asm volatile("cp.async.wait_group 0;" ::: "memory");
  else if (n == 1) asm volatile("cp.async.wait_group 1;" ::: "memory");
  else asm volatile("cp.async.wait_group 2;" ::: "memory");
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// Bias (and GELU) on this thread's row of 64 accumulators (columns n..n+63),
// packed into 32 bf16 pairs.
template <Epi E>
__device__ __forceinline__ void bias_act_pack64(const EpiArgs& ea, int n, const uint32_t (&acc)[2][32],
                                                uint32_t (&wv)[32]) {
  const uint4* bias4 = reinterpret_cast<const uint4*>(static_cast<const bf16*>(ea.bias) + n);
#pragma unroll
  for (int q = 0; q < 8; ++q) {
    const uint4 bq = __ldg(bias4 + q);
    const uint32_t bw[4] = {bq.x, bq.y, bq.z, bq.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int c0 = 8 * q + 2 * j;
      float v0 = __uint_as_float(acc[c0 / 32][c0 % 32]) + bf16_lo(bw[j]);
      float v1 = __uint_as_float(acc[(c0 + 1) / 32][(c0 + 1) % 32]) + bf16_hi(bw[j]);
      if constexpr (E == Epi::BiasGelu) gelu2_as7126(v0, v1);
      wv[4 * q + j] = pack_bf16x2(v0, v1);
    }
  }
}

// bf16 epilogues (bias; bias + GELU) over W = 64 or 32 consecutive columns
// n..n+W-1 of the warp's 32 rows row0..row0+31: each thread biases (and GELUs)
// its own row and packs it into W/2 bf16 pairs in shared memory, then the warp
// writes the chunk row by row, so every store covers 2W contiguous bytes.
template <Epi E, int W>
__device__ __forceinline__ void epilogue_bf16(const EpiArgs& ea, int row0, int M, int n, int N,
                                              const uint32_t (&acc)[W / 32][32], uint32_t* stg,
                                              int lane) {
  const uint4* bias4 = reinterpret_cast<const uint4*>(static_cast<const bf16*>(ea.bias) + n);
#pragma unroll
  for (int q = 0; q < W / 8; ++q) {
    const uint4 bq = __ldg(bias4 + q);
    const uint32_t bw[4] = {bq.x, bq.y, bq.z, bq.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int c0 = 8 * q + 2 * j;
      float v0 = __uint_as_float(acc[c0 / 32][c0 % 32]) + bf16_lo(bw[j]);
      float v1 = __uint_as_float(acc[(c0 + 1) / 32][(c0 + 1) % 32]) + bf16_hi(bw[j]);
      if constexpr (E == Epi::BiasGelu) gelu2_as7126(v0, v1);
      stg[lane * 33 + 4 * q + j] = pack_bf16x2(v0, v1);
    }
  }
  __syncwarp();
  uint32_t* out = static_cast<uint32_t*>(ea.out);        // bf16 pairs
  const int ldw = N / 2;
  if constexpr (W == 64) {
#pragma unroll 8
    for (int i = 0; i < 32; ++i)
      if (row0 + i < M) out[size_t(row0 + i) * ldw + n / 2 + lane] = stg[i * 33 + lane];
  } else {
    // 16 pairs per row: half a warp per row, two rows per store
#pragma unroll 8
    for (int i = 0; i < 32; i += 2) {
      const int rr = i + (lane >> 4);
      if (row0 + rr < M)
        out[size_t(row0 + rr) * ldw + n / 2 + (lane & 15)] = stg[rr * 33 + (lane & 15)];
    }
  }
  __syncwarp();
}

// Residual epilogues through a per-warp shared-memory transpose: the warp's 32
// rows x 32 columns of accumulators go to shared memory row by row (one row per
// thread), then each thread takes one column and the warp walks the 32 rows, so
// every fp32 load and store of the residual stream covers 128 contiguous bytes.
// row0: first tile row of this warp; n: first column of the chunk.
// The residual rows of a chunk, one column per thread (loads issued together).
__device__ __forceinline__ void load_residual(const EpiArgs& ea, int row0, int M, int n, int N,
                                              int lane, float (&rv)[32]) {
#pragma unroll
  for (int i = 0; i < 32; ++i)
    rv[i] = row0 + i < M ? ea.res[size_t(row0 + i) * N + n + lane] : 0.f;
}

template <Epi E>
__device__ __forceinline__ void epilogue32_rows(const EpiArgs& ea, int row0, int M, int n, int N,
                                                const uint32_t (&acc)[32], const float (&rv)[32],
                                                float* stg, int lane) {
#pragma unroll
  for (int j = 0; j < 32; ++j) stg[lane * 33 + j] = __uint_as_float(acc[j]);
  __syncwarp();
  const int col = n + lane;
  const float bias = __bfloat162float(static_cast<const bf16*>(ea.bias)[col]);
  float* out = static_cast<float*>(ea.out);
  // the residual of the chunk was loaded before (the update is in place)
  if constexpr (E == Epi::BiasResidual) {
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if (row0 + i < M) out[size_t(row0 + i) * N + col] = rv[i] + (stg[i * 33 + lane] + bias);
  } else {
    // last sparse block: hn = h + f(h); x'[xrow] = x0 + (hn - h0), h0 == x0.
    // Element offsets fit 32 bits: sr_create rejects B * L * width >= 2^31.
#pragma unroll
    for (int half = 0; half < 32; half += 16) {
      uint32_t xrow[16];
      float x0[16];
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        const int m = row0 + half + i < M ? row0 + half + i : row0;
        xrow[i] = (uint32_t(m / ea.Kr) * uint32_t(ea.Lx) + uint32_t(ea.idx[m])) * uint32_t(N) +
                  uint32_t(col);
      }
#pragma unroll
      for (int i = 0; i < 16; ++i) x0[i] = row0 + half + i < M ? out[xrow[i]] : 0.f;
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        if (row0 + half + i < M) {
          const float hn = rv[half + i] + (stg[(half + i) * 33 + lane] + bias);
          out[xrow[i]] = x0[i] + (hn - x0[i]);
        }
      }
    }
  }
  __syncwarp();
}

template <int BN, Epi E, bool kPair>
__global__ void __launch_bounds__(kThreads, 1)
gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
               const __grid_constant__ CUtensorMap tmR, int M, int N, int K, EpiArgs ea) {
  using C = GemmCfg<BN, E, kPair>;
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* base = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* sA = base;
  unsigned char* sB = base + size_t(C::kStages) * C::kABytes;
  float* staging = reinterpret_cast<float*>(base + size_t(C::kStages) * C::kStageBytes);
  Smem* sm = reinterpret_cast<Smem*>(base + size_t(C::kStages) * C::kStageBytes +
                                     C::kStagingBytes);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int m_tiles = (M + C::kRowsTile - 1) / C::kRowsTile;
  const int n_tiles = N / BN;
  const int tiles = m_tiles * n_tiles;
  const int kblocks = K / BK;
  // a pair works through the tiles as one unit; rank 1 holds rows 128..255
  const uint32_t rank = kPair ? cluster_ctarank() : 0u;
  const int unit = kPair ? int(blockIdx.x >> 1) : int(blockIdx.x);
  const int units = kPair ? int(gridDim.x >> 1) : int(gridDim.x);

  if (threadIdx.x == 0) {
    // a pair's stage is full once both producers announced their bytes and they
    // landed; its accumulator is free once both epilogues have read it
    for (int s = 0; s < C::kStages; ++s) { mbar_init(&sm->full[s], kPair ? 2 : 1); mbar_init(&sm->empty[s], 1); }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&sm->tfull[a], 1);
      mbar_init(&sm->tempty[a], kPair ? 2 * (kEpiThreads / 32) : kEpiThreads);   // a pair: one per warp
    }
    mbar_init(&sm->drain, 1);
    for (int w = 0; w < kEpiThreads / 32; ++w) { mbar_init(&sm->res_full[w][0], 1); mbar_init(&sm->res_full[w][1], 1); }
    sm->abort = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
    if constexpr (C::kTmaRes || C::kTmaOut) prefetch_tmap(&tmR);
  }
  if (warp == 1) {
    if constexpr (kPair) tmem_alloc_pair(&sm->tmem_base, C::kTmemCols);
    else tmem_alloc(&sm->tmem_base, C::kTmemCols);
  }
  tc_fence_before();
  if constexpr (kPair) cluster_sync();   // both CTAs' barriers exist before any remote arrival
  else __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm->tmem_base;
  volatile int* abort = &sm->abort;
  if (warp == 0 && lane == 0 && unit < tiles) {
    // the weights do not depend on the previous kernel: the first tile's weight
    // rows start moving into L2 while it finishes
    const int brow = (unit % n_tiles) * BN + int(rank) * C::kBRows;
    for (int kb = 0; kb < kblocks; ++kb) tma_prefetch_l2_2d(&tmB, kb * BK, brow);
  }
  pdl_wait();      // the previous kernel's writes are visible from here
  pdl_trigger();
  // an abort in one CTA of a pair stops the other's waits too
  auto abort_peer = [&]() {
    if constexpr (kPair) {
      if (*abort) st_cluster_u32(mapa_shared(&sm->abort, rank ^ 1u), 1u);
    }
  };

  if (warp == 0) {
    // ---------------------------------------------------------- TMA producer
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued = 0, issued_phase = 0;    // per stage: loads in flight, their parity
      // a pair's loads complete on the even CTA's full barrier
      const uint32_t full0 = kPair ? mapa_shared(&sm->full[0], 0) : 0u;
      for (int t = unit; t < tiles && !*abort; t += units) {
        const int nt = t % n_tiles, mt = t / n_tiles;
        const int arow = mt * C::kRowsTile + int(rank) * BM;
        const int brow = nt * BN + int(rank) * C::kBRows;
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait<kPair>(&sm->empty[stage], phase ^ 1, abort, ea.fault)) break;
          if constexpr (kPair) {
            const uint32_t fb = full0 + uint32_t(stage) * 8u;
            mbar_arrive_expect_tx_relaxed_cluster(fb, C::kStageBytes);
            tma_load_2d_pair(&tmA, sA + size_t(stage) * C::kABytes, fb, kb * BK, arow);
            tma_load_2d_pair(&tmB, sB + size_t(stage) * C::kBBytes, fb, kb * BK, brow);
          } else {
            mbar_arrive_expect_tx(&sm->full[stage], C::kStageBytes);
            tma_load_2d(&tmA, sA + size_t(stage) * C::kABytes, &sm->full[stage], kb * BK, arow);
            tma_load_2d(&tmB, sB + size_t(stage) * C::kBBytes, &sm->full[stage], kb * BK, brow);
          }
          issued |= 1u << stage;
          issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
          if (++stage == C::kStages) { stage = 0; phase ^= 1; }
        }
      }
      abort_peer();
      // every load this thread issued lands before the CTA may exit (immediate
      // unless an aborted pipeline left loads unconsumed); a pair's loads are
      // counted on the even CTA's barriers, which its MMA thread drains
      int no_abort = 0;
      if constexpr (!kPair) {
        for (int st = 0; st < C::kStages; ++st)
          if (issued & (1u << st)) mbar_wait(&sm->full[st], (issued_phase >> st) & 1u, &no_abort, ea.fault);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------------------- MMA issuer
    // (of a pair, only the even CTA issues; its commits arrive in both CTAs)
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = idesc_bf16(C::kRowsTile, BN);
      int stage = 0;
      uint32_t phase = 0;
      int it = 0;
      for (int t = unit; t < tiles && !*abort; t += units, ++it) {
        const int acc = it & 1;
        const uint32_t aphase = (it >> 1) & 1;
        if (!mbar_wait<kPair>(&sm->tempty[acc], aphase ^ 1, abort, ea.fault)) break;
        tc_fence_after();
        const uint32_t d = tmem + uint32_t(acc * BN);
        for (int kb = 0; kb < kblocks; ++kb) {
          if (!mbar_wait<kPair>(&sm->full[stage], phase, abort, ea.fault)) break;
          tc_fence_after();
          const uint32_t a0 = smem_u32(sA + size_t(stage) * C::kABytes);
          const uint32_t b0 = smem_u32(sB + size_t(stage) * C::kBBytes);
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            if constexpr (kPair)
              mma_bf16_pair(d, sw128_desc(a0 + 32 * k), sw128_desc(b0 + 32 * k), idesc,
                            (kb | k) != 0 ? 1u : 0u);
            else
              mma_bf16(d, sw128_desc(a0 + 32 * k), sw128_desc(b0 + 32 * k), idesc,
                       (kb | k) != 0 ? 1u : 0u);
          }
          if constexpr (kPair) mma_commit_pair_both(&sm->empty[stage]);
          else mma_commit(&sm->empty[stage]);
          if (++stage == C::kStages) { stage = 0; phase ^= 1; }
        }
        if constexpr (kPair) mma_commit_pair_both(&sm->tfull[acc]);
        else mma_commit(&sm->tfull[acc]);
      }
      abort_peer();
      // every MMA issued has completed before the tensor memory is released
      int no_abort = 0;
      if constexpr (kPair) mma_commit_pair_local(&sm->drain);
      else mma_commit(&sm->drain);
      mbar_wait(&sm->drain, 0, &no_abort, ea.fault);
    }
  } else {
    // ---------------------------------------------------------- epilogue
    const int q = warp & 3;                 // TMEM lane quarter of this warp
    const int half = (warp - 2) >> 2;       // which half of the tile's columns
    constexpr int kW = BN / 2 >= 64 ? 64 : 32;    // bf16 epilogue step (columns)
    int it = 0;
    const uint32_t tempty0 = kPair ? mapa_shared(&sm->tempty[0], 0) : 0u;
    for (int t = unit; t < tiles; t += units, ++it) {
      const int nt = t % n_tiles, mt = t / n_tiles;
      const int acc = it & 1;
      const uint32_t aphase = (it >> 1) & 1;
      const int row0 = mt * C::kRowsTile + int(rank) * BM + q * 32;
      const int c_begin = half * (BN / 2), c_end = (half + 1) * (BN / 2);
      if constexpr (C::kTmaOut) {
        if (!__all_sync(0xffffffffu, mbar_wait<kPair>(&sm->tfull[acc], aphase, abort, ea.fault))) break;
        tc_fence_after();
        const uint32_t tbase = tmem + (uint32_t(q * 32) << 16) + uint32_t(acc * BN);
        unsigned char* obuf = reinterpret_cast<unsigned char*>(staging) +
                              size_t(warp - 2) * C::kOutTileBytes;
#pragma unroll 1
        for (int c = c_begin; c < c_end; c += 64) {
          uint32_t r[2][32];
          tmem_ld32(tbase + uint32_t(c), r[0]);
          tmem_ld32(tbase + uint32_t(c + 32), r[1]);
          tmem_wait_ld();
          uint32_t wv[32];
          bias_act_pack64<E>(ea, nt * BN + c, r, wv);
          // the previous store from this buffer has read it before it is rewritten
          if (lane == 0) bulk_wait_read_all();
          __syncwarp();
          // this thread's row: 16-byte chunk j of the row sits at slot j ^ (row % 8)
          uint4* rowp = reinterpret_cast<uint4*>(obuf + lane * 128);
#pragma unroll
          for (int j = 0; j < 8; ++j)
            rowp[j ^ (lane & 7)] = make_uint4(wv[4 * j], wv[4 * j + 1], wv[4 * j + 2], wv[4 * j + 3]);
          fence_proxy_async_smem();
          __syncwarp();
          // rows past M are clipped by the tensor map
          if (lane == 0 && row0 < M) {
            tma_store_2d(&tmR, obuf, nt * BN + c, row0);
            bulk_commit_group();
          }
        }
      } else if constexpr (E == Epi::Bias || E == Epi::BiasGelu) {
        if (!__all_sync(0xffffffffu, mbar_wait<kPair>(&sm->tfull[acc], aphase, abort, ea.fault))) break;
        tc_fence_after();
        const uint32_t tbase = tmem + (uint32_t(q * 32) << 16) + uint32_t(acc * BN);
#pragma unroll 1
        for (int c = c_begin; c < c_end; c += kW) {
          uint32_t r[kW / 32][32];
#pragma unroll
          for (int k = 0; k < kW / 32; ++k) tmem_ld32(tbase + uint32_t(c + 32 * k), r[k]);
          tmem_wait_ld();
          epilogue_bf16<E, kW>(ea, row0, M, nt * BN + c, N, r,
                               reinterpret_cast<uint32_t*>(staging) + (warp - 2) * C::kStageFloats,
                               lane);
        }
      } else if constexpr (C::kTmaRes) {
        // residual tiles by TMA: the warp's half of the tile's columns is walked in
        // 32-column chunks (32 rows x 32 fp32, 128-byte swizzle) through two
        // buffers; the first two are requested before the accumulator is ready,
        // each chunk is updated in place and stored back by TMA, and a buffer is
        // refilled once its store has read it
        constexpr int kChunks = BN / 64;
        static_assert(kChunks % 2 == 0, "chunks alternate between two buffers");
        unsigned char* rbuf = reinterpret_cast<unsigned char*>(staging) +
                              size_t(warp - 2) * 2 * C::kResTileBytes;
        uint64_t* rbar = sm->res_full[warp - 2];
        if (!ea.sqnorm) {
          // bias + accumulator staged per chunk and added into the stream by TMA
          // reduce: the residual itself never passes through the SM
          if (!__all_sync(0xffffffffu, mbar_wait<kPair>(&sm->tfull[acc], aphase, abort, ea.fault))) break;
          tc_fence_after();
          const uint32_t tbase = tmem + (uint32_t(q * 32) << 16) + uint32_t(acc * BN);
#pragma unroll 1
          for (int k = 0; k < kChunks; ++k) {
            const int c = c_begin + 32 * k;
            uint32_t r[32];
            tmem_ld32(tbase + uint32_t(c), r);
            tmem_wait_ld();
            // the buffer's previous reduce (two chunks back) has read it
            if (lane == 0) bulk_wait_read_le1();
            __syncwarp();
            float4* rowp = reinterpret_cast<float4*>(rbuf + (k & 1) * C::kResTileBytes + lane * 128);
            const uint4* bias4 =
                reinterpret_cast<const uint4*>(static_cast<const bf16*>(ea.bias) + nt * BN + c);
#pragma unroll
            for (int jq = 0; jq < 4; ++jq) {
              const uint4 bq = __ldg(bias4 + jq);
              const uint32_t bw[4] = {bq.x, bq.y, bq.z, bq.w};
#pragma unroll
              for (int h2 = 0; h2 < 2; ++h2) {
                const int j = 2 * jq + h2;
                rowp[j ^ (lane & 7)] =
                    make_float4(__uint_as_float(r[4 * j]) + bf16_lo(bw[2 * h2]),
                                __uint_as_float(r[4 * j + 1]) + bf16_hi(bw[2 * h2]),
                                __uint_as_float(r[4 * j + 2]) + bf16_lo(bw[2 * h2 + 1]),
                                __uint_as_float(r[4 * j + 3]) + bf16_hi(bw[2 * h2 + 1]));
              }
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0 && row0 < M) {
              tma_reduce_add_2d(&tmR, rbuf + (k & 1) * C::kResTileBytes, nt * BN + c, row0);
              bulk_commit_group();
            }
          }
        } else {
        auto request = [&](int k) {   // lane 0 only
          mbar_arrive_expect_tx(&rbar[k & 1], C::kResTileBytes);
          tma_load_2d(&tmR, rbuf + (k & 1) * C::kResTileBytes, &rbar[k & 1],
                      nt * BN + c_begin + 32 * k, row0);
        };
        // parity of chunk k's buffer barrier: each barrier completes kChunks / 2 times a tile
        auto parity = [&](int k) { return uint32_t(it * (kChunks / 2) + (k >> 1)) & 1u; };
        if (lane == 0) {
          bulk_wait_read_all();          // the previous tile's stores left both buffers
          request(0);
          request(1);
          // the later chunks move into L2 while the tile's mainloop runs: a launch
          // whose tiles end together would otherwise stream the whole residual
          // stream from HBM in its tail
          if (row0 < M)
            for (int k = 2; k < kChunks; ++k) tma_prefetch_l2_2d(&tmR, nt * BN + c_begin + 32 * k, row0);
        }
        int consumed = 0, requested = 2;
        float sq = 0.f;                  // this thread's row: squares of the bf16-rounded update
        bool ok = __all_sync(0xffffffffu, mbar_wait<kPair>(&sm->tfull[acc], aphase, abort, ea.fault));
        if (ok) {
          tc_fence_after();
          const uint32_t tbase = tmem + (uint32_t(q * 32) << 16) + uint32_t(acc * BN);
#pragma unroll 1
          for (int k = 0; k < kChunks && ok; ++k) {
            const int c = c_begin + 32 * k;
            uint32_t r[32];
            tmem_ld32(tbase + uint32_t(c), r);
            tmem_wait_ld();
            if (!(ok = __all_sync(0xffffffffu, mbar_wait(&rbar[k & 1], parity(k), abort, ea.fault)))) break;
            consumed = k + 1;
            // this thread's row: 16-byte chunk j of the row sits at slot j ^ (row % 8)
            float4* rowp = reinterpret_cast<float4*>(rbuf + (k & 1) * C::kResTileBytes + lane * 128);
            const uint4* bias4 =
                reinterpret_cast<const uint4*>(static_cast<const bf16*>(ea.bias) + nt * BN + c);
#pragma unroll
            for (int jq = 0; jq < 4; ++jq) {
              const uint4 bq = __ldg(bias4 + jq);
              const uint32_t bw[4] = {bq.x, bq.y, bq.z, bq.w};
#pragma unroll
              for (int h2 = 0; h2 < 2; ++h2) {
                const int j = 2 * jq + h2;
                float4 v = rowp[j ^ (lane & 7)];
                v.x += __uint_as_float(r[4 * j]) + bf16_lo(bw[2 * h2]);
                v.y += __uint_as_float(r[4 * j + 1]) + bf16_hi(bw[2 * h2]);
                v.z += __uint_as_float(r[4 * j + 2]) + bf16_lo(bw[2 * h2 + 1]);
                v.w += __uint_as_float(r[4 * j + 3]) + bf16_hi(bw[2 * h2 + 1]);
                rowp[j ^ (lane & 7)] = v;
                if (ea.sqnorm) {
                  const float q4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                  for (int e = 0; e < 4; ++e) {
                    const float rq = __bfloat162float(__float2bfloat16_rn(q4[e]));
                    sq = fmaf(rq, rq, sq);
                  }
                }
              }
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              if (row0 < M) {
                tma_store_2d(&tmR, rbuf + (k & 1) * C::kResTileBytes, nt * BN + c, row0);
                bulk_commit_group();
              }
              if (k + 2 < kChunks) {
                bulk_wait_read_all();    // this chunk's store has read the buffer
                request(k + 2);
              }
            }
            if (k + 2 < kChunks) requested = k + 3;
          }
        }
        // one partial sum per row and half tile, in its own slot (the sum over the
        // slots is taken in a fixed order, so the scores are reproducible)
        if (ok && ea.sqnorm && row0 + lane < M)
          ea.sqnorm[size_t(row0 + lane) * (2 * n_tiles) + (nt * 2 + half)] = sq;
        if (!ok) {
          // an aborted pipeline: the residual loads requested above still land first
          int no_abort = 0;
          if (lane == 0)
            for (int k = consumed; k < requested; ++k)
              mbar_wait(&rbar[k & 1], parity(k), &no_abort, ea.fault);
          __syncwarp();
          break;
        }
        }
      } else if constexpr (E == Epi::BiasResidualScatter) {
        // last sparse block: hn = h + f(h); x'[xrow] = x0 + (hn - x0), h0 == x0.
        // Every row the warp reads (the routed rows h and the stream rows x0
        // they scatter into, 128 contiguous bytes per row and 32 columns) is
        // prefetched into L2 while the mainloop runs.  On the unit's last tile
        // the rows are then copied into the idle operand ring, three 32-column
        // quarters at once; on earlier tiles (the ring is still in use) the warp
        // walks its 32 rows x BN/2 columns in steps of 16 rows x 32 columns with
        // each step's loads issued one step ahead.  Either way a thread owns one
        // column of a row at a time (through the per-warp transpose buffer), so
        // every store of a row covers 128 contiguous bytes, and the arithmetic is
        // the same.  Element offsets fit 32 bits: sr_create rejects B * L *
        // width >= 2^31.
        constexpr int kSteps = 2 * (BN / 64);
        const int m_lane = row0 + lane;
        const uint32_t xrow_lane =
            m_lane < M ? (uint32_t(m_lane / ea.Kr) * uint32_t(ea.Lx) + uint32_t(__ldg(ea.idx + m_lane))) *
                             uint32_t(N)
                       : 0u;
        const float* hres = ea.res;
        float* xs = static_cast<float*>(ea.out);
        // step st: columns c_begin + 32 (st / 2) .. + 31, rows 16 (st % 2) .. + 15
        auto load_step = [&](int st, float (&h)[16], float (&x)[16]) {
          const int n = nt * BN + c_begin + 32 * (st >> 1) + lane;
          const int i0 = 16 * (st & 1);
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const uint32_t xr = __shfl_sync(0xffffffffu, xrow_lane, i0 + i);
            const bool v = row0 + i0 + i < M;
            h[i] = v ? hres[size_t(row0 + i0 + i) * N + n] : 0.f;
            x[i] = v ? xs[xr + uint32_t(n)] : 0.f;
          }
        };
        // every row this warp reads moves into L2 while the tile's mainloop runs
        if (m_lane < M) {
          const char* hp = reinterpret_cast<const char*>(hres + size_t(m_lane) * N + nt * BN + c_begin);
          const char* xp = reinterpret_cast<const char*>(xs + xrow_lane + uint32_t(nt * BN + c_begin));
#pragma unroll
          for (int l = 0; l < BN / 2 * 4 / 128; ++l) {
            prefetch_l2(hp + 128 * l);
            prefetch_l2(xp + 128 * l);
          }
        }
        if (t + units >= tiles) {
          // the unit's last tile: once the accumulator is ready no MMA reads the
          // operand ring and no load refills it, so each warp stages there the
          // rows it updates, a 32-column quarter at a time (its routed rows h
          // and the stream rows x0), with up to three quarters in flight
          if (!__all_sync(0xffffffffu, mbar_wait<kPair>(&sm->tfull[acc], aphase, abort, ea.fault))) break;
          tc_fence_after();
          fence_proxy_async_smem();      // the ring was last written and read by the async proxy
          unsigned char* wbuf = sA + size_t(warp - 2) * C::kScatterSlots * C::kScatterSlotBytes;
          auto fetch = [&](int k) {
            unsigned char* hb = wbuf + (k % C::kScatterSlots) * C::kScatterSlotBytes;
            const int col = nt * BN + c_begin + 32 * k + 4 * (lane & 7);
#pragma unroll
            for (int rr = 0; rr < 8; ++rr) {
              const int i = (lane >> 3) + 4 * rr;      // 4 rows x 128 bytes per instruction
              const uint32_t xr = __shfl_sync(0xffffffffu, xrow_lane, i);
              if (row0 + i < M) {
                cp_async16(hb + i * 128 + (lane & 7) * 16, hres + size_t(row0 + i) * N + col);
                cp_async16(hb + 4096 + i * 128 + (lane & 7) * 16, xs + xr + uint32_t(col));
              }
            }
            cp_async_commit();
          };
#pragma unroll
          for (int k = 0; k < C::kScatterSlots; ++k) fetch(k);
          const uint32_t tbase = tmem + (uint32_t(q * 32) << 16) + uint32_t(acc * BN);
          float* stg = staging + (warp - 2) * C::kStageFloats;
#pragma unroll 1
          for (int k = 0; k < C::kScatterQuarters; ++k) {
            const int c = c_begin + 32 * k;
            uint32_t r[32];
            tmem_ld32(tbase + uint32_t(c), r);
            tmem_wait_ld();
#pragma unroll
            for (int j = 0; j < 32; ++j) stg[lane * 33 + j] = __uint_as_float(r[j]);
            // quarter k has landed once at most the later ones are in flight
            const int issued = min(C::kScatterQuarters, k + C::kScatterSlots);
            cp_async_wait_upto(issued - (k + 1));
            __syncwarp();
            const float* hq =
                reinterpret_cast<const float*>(wbuf + (k % C::kScatterSlots) * C::kScatterSlotBytes);
            const float* xq = hq + 32 * 32;
            const int col = nt * BN + c + lane;
            const float bias = __bfloat162float(static_cast<const bf16*>(ea.bias)[col]);
#pragma unroll 4
            for (int i = 0; i < 32; ++i) {
              const uint32_t xr = __shfl_sync(0xffffffffu, xrow_lane, i);
              if (row0 + i < M) {
                const float hn = hq[i * 32 + lane] + (stg[i * 33 + lane] + bias);
                const float x0v = xq[i * 32 + lane];
                xs[xr + uint32_t(col)] = x0v + (hn - x0v);
              }
            }
            __syncwarp();                // the slot and the transpose buffer are rewritten next
            if (k + C::kScatterSlots < C::kScatterQuarters) fetch(k + C::kScatterSlots);
          }
        } else {
          float rv[2][16], x0[2][16];
          load_step(0, rv[0], x0[0]);
          if (!__all_sync(0xffffffffu, mbar_wait<kPair>(&sm->tfull[acc], aphase, abort, ea.fault))) break;
          tc_fence_after();
          const uint32_t tbase = tmem + (uint32_t(q * 32) << 16) + uint32_t(acc * BN);
          float* stg = staging + (warp - 2) * C::kStageFloats;
#pragma unroll
          for (int st = 0; st < kSteps; ++st) {
            const int c = c_begin + 32 * (st >> 1);
            if ((st & 1) == 0) {
              // this thread's row of the chunk's accumulators into the transpose buffer
              uint32_t r[32];
              tmem_ld32(tbase + uint32_t(c), r);
              tmem_wait_ld();
#pragma unroll
              for (int j = 0; j < 32; ++j) stg[lane * 33 + j] = __uint_as_float(r[j]);
              __syncwarp();
            }
            if (st + 1 < kSteps) load_step(st + 1, rv[(st + 1) & 1], x0[(st + 1) & 1]);
            const int col = nt * BN + c + lane;
            const float bias = __bfloat162float(static_cast<const bf16*>(ea.bias)[col]);
            const int i0 = 16 * (st & 1);
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              const uint32_t xr = __shfl_sync(0xffffffffu, xrow_lane, i0 + i);
              if (row0 + i0 + i < M) {
                const float hn = rv[st & 1][i] + (stg[(i0 + i) * 33 + lane] + bias);
                xs[xr + uint32_t(col)] = x0[st & 1][i] + (hn - x0[st & 1][i]);
              }
            }
            if (st & 1) __syncwarp();      // the next chunk rewrites the transpose buffer
          }
        }
      } else {
        // the first chunk's residual loads overlap the wait for the accumulator
        float rv[32];
        load_residual(ea, row0, M, nt * BN + c_begin, N, lane, rv);
        if (!__all_sync(0xffffffffu, mbar_wait<kPair>(&sm->tfull[acc], aphase, abort, ea.fault))) break;
        tc_fence_after();
        const uint32_t tbase = tmem + (uint32_t(q * 32) << 16) + uint32_t(acc * BN);
#pragma unroll 1
        for (int c = c_begin; c < c_end; c += 32) {
          uint32_t r[32];
          tmem_ld32(tbase + uint32_t(c), r);
          tmem_wait_ld();
          epilogue32_rows<E>(ea, row0, M, nt * BN + c, N, r, rv,
                             staging + (warp - 2) * C::kStageFloats, lane);
          if (c + 32 < c_end) load_residual(ea, row0, M, nt * BN + c + 32, N, lane, rv);
        }
      }
      tc_fence_before();
      if constexpr (kPair) {
        __syncwarp();
        if (lane == 0) {
          if (rank == 0) mbar_arrive(&sm->tempty[acc]);
          else mbar_arrive_cluster(tempty0 + uint32_t(acc) * 8u);
        }
      } else {
        mbar_arrive(&sm->tempty[acc]);
      }
    }
    if (lane == 0) abort_peer();
    if constexpr (C::kTmaRes || C::kTmaOut) {
      // the TMA stores have read shared memory before the CTA exits; their
      // writes are complete when the grid is
      if (lane == 0) bulk_wait_read_all();
    }
  }
  tc_fence_before();
  if constexpr (kPair) cluster_sync();   // neither CTA leaves while the other may still signal it
  else __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    if constexpr (kPair) tmem_dealloc_pair(tmem, C::kTmemCols);
    else tmem_dealloc(tmem, C::kTmemCols);
  }
}

// ------------------------------------------------------------------ host side
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

cudaError_t get_encoder() {
  if (g_encode) return cudaSuccess;
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                   cudaEnableDefault, &q);
  if (e != cudaSuccess) return e;
  if (q != cudaDriverEntryPointSuccess || !fn) return cudaErrorNotSupported;
  g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  return cudaSuccess;
}

// 2-D bf16 tensor map over a row-major [rows, cols] matrix, box [box_rows, 64].
cudaError_t make_map_2d(CUtensorMap* map, const void* ptr, uint64_t rows, uint64_t cols,
                        uint32_t box_rows) {
  cudaError_t e = get_encoder();
  if (e != cudaSuccess) return e;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}


// 2-D fp32 tensor map over a row-major [rows, cols] matrix, box [32, 32],
// 128-byte swizzle (the residual stream tiles of the TMA epilogue).
cudaError_t make_map_f32_32x32(CUtensorMap* map, const void* ptr, uint64_t rows, uint64_t cols) {
  cudaError_t e = get_encoder();
  if (e != cudaSuccess) return e;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 4};
  cuuint32_t box[2] = {32, 32};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(ptr), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

template <int BN, Epi E, bool kPair>
cudaError_t launch_bn(const void* A, const void* W, int M, int N, int K, const EpiArgs& ea,
                      cudaStream_t s) {
  using C = GemmCfg<BN, E, kPair>;
  CUtensorMap ta, tb, tr;
  cudaError_t e = make_map_2d(&ta, A, uint64_t(M), uint64_t(K), BM);
  if (e != cudaSuccess) return e;
  e = make_map_2d(&tb, W, uint64_t(N), uint64_t(K), C::kBRows);
  if (e != cudaSuccess) return e;
  if constexpr (C::kTmaRes) {
    // the update is in place: the residual read and the output are one tensor
    if (ea.res != ea.out) return cudaErrorInvalidValue;
    e = make_map_f32_32x32(&tr, ea.out, uint64_t(M), uint64_t(N));
    if (e != cudaSuccess) return e;
  } else if constexpr (C::kTmaOut) {
    e = make_map_2d(&tr, ea.out, uint64_t(M), uint64_t(N), 32);   // box 32 rows x 64 columns
    if (e != cudaSuccess) return e;
  } else {
    tr = tb;    // unused
  }
  auto kernel = gemm_tc_kernel<BN, E, kPair>;
  // CTAs (or CTA pairs) resident at once, per device
  static int max_units_of[kMaxDevices] = {};
  const int slot = device_slot();
  if (slot < 0) return cudaErrorInvalidDevice;
  int& max_units = max_units_of[slot];
  if (max_units == 0) {
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(C::kSmem));
    if (e != cudaSuccess) return e;
    int num_sms = 0;
    e = cudaDeviceGetAttribute(&num_sms, cudaDevAttrMultiProcessorCount, slot);
    if (e != cudaSuccess) return e;
    if constexpr (kPair) {
      cudaLaunchConfig_t cfg = {};
      cudaLaunchAttribute at[1];
      at[0].id = cudaLaunchAttributeClusterDimension;
      at[0].val.clusterDim.x = 2; at[0].val.clusterDim.y = 1; at[0].val.clusterDim.z = 1;
      cfg.gridDim = dim3(unsigned(num_sms & ~1));
      cfg.blockDim = dim3(kThreads);
      cfg.dynamicSmemBytes = C::kSmem;
      cfg.attrs = at;
      cfg.numAttrs = 1;
      int clusters = 0;
      e = cudaOccupancyMaxActiveClusters(&clusters, kernel, &cfg);
      if (e != cudaSuccess) return e;
      if (clusters < 1) return cudaErrorInvalidConfiguration;
      max_units = clusters;
    } else {
      max_units = num_sms;
    }
  }
  const int tiles = ((M + C::kRowsTile - 1) / C::kRowsTile) * (N / BN);
  const int units = tiles < max_units ? tiles : max_units;
  return launch_k(kernel, dim3(unsigned(kPair ? 2 * units : units)), dim3(kThreads), C::kSmem, s,
                  kPair ? 2u : 1u, ta, tb, tr, M, N, K, ea);
}

template <int BN, bool kPair>
cudaError_t launch_epi(Epi epi, const void* A, const void* W, int M, int N, int K,
                       const EpiArgs& ea, cudaStream_t s) {
  switch (epi) {
    case Epi::Bias: return launch_bn<BN, Epi::Bias, kPair>(A, W, M, N, K, ea, s);
    case Epi::BiasGelu: return launch_bn<BN, Epi::BiasGelu, kPair>(A, W, M, N, K, ea, s);
    case Epi::BiasResidualScatter:
      return launch_bn<BN, Epi::BiasResidualScatter, kPair>(A, W, M, N, K, ea, s);
    case Epi::BiasResidual:   // chosen in launch_gemm_tc
      break;
  }
  return cudaErrorInvalidValue;
}

}  // namespace

int gemm_tc_sqnorm_parts(int N) {
  // BiasResidual runs 256-column pair tiles when 256 divides N, else 128-column ones
  if (N % 256 == 0) return N / 128;
  if (N % 128 == 0) return N / 64;
  return 0;
}

cudaError_t launch_gemm_tc(Epi epi, const void* A, const void* W, int M, int N, int K,
                           const EpiArgs& ea, cudaStream_t s) {
  if (M < 1 || K % BK != 0 || N % 64 != 0) return cudaErrorInvalidValue;
  if (ea.sqnorm && (epi != Epi::BiasResidual || gemm_tc_sqnorm_parts(N) == 0)) return cudaErrorInvalidValue;
  // tiles 128 or 256 columns wide run on CTA pairs (256-row tiles); 64-wide on single CTAs
  if (epi == Epi::BiasResidual) {
    // pair tiles update the fp32 residual stream through the TMA epilogue
    if (N % 256 == 0) return launch_bn<256, Epi::BiasResidual, true>(A, W, M, N, K, ea, s);
    if (N % 128 == 0) return launch_bn<128, Epi::BiasResidual, true>(A, W, M, N, K, ea, s);
    return launch_bn<64, Epi::BiasResidual, false>(A, W, M, N, K, ea, s);
  }
  if (N % 256 == 0) return launch_epi<256, true>(epi, A, W, M, N, K, ea, s);
  if (N % 128 == 0) return launch_epi<128, true>(epi, A, W, M, N, K, ea, s);
  return launch_epi<64, false>(epi, A, W, M, N, K, ea, s);
}

}  // namespace sr
