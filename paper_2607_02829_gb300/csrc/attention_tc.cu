// tcgen05 flash attention for head_dim 64, bf16 q/k/v, fp32 softmax statistics:
// out[b, t, h*64 : h*64+64] = softmax(q k^T / 8) v over the T tokens of sample b
// (the attention of the pre-LN block, Sec. 3.3 Eq. 11; within the sparse stage
// T = K and the tokens are the routed ones, Eq. 8).  No mask; keys beyond T in
// the last tile are excluded.
//
// One CTA owns 256 query rows of one (sample, head) as two 128-row tiles that
// share every K/V tile, 384 threads:
//   warp 0      TMA: the two Q tiles once, then K_j and V_j, 128 keys x 64, into
//               two 3-stage rings (3-D tensor map over [B, T, 3D], zero fill
//               past T); a K stage frees as soon as both tiles' S MMAs that read
//               it finish, a V stage when both tiles' P V MMAs do;
//   warp 1      issues S^t = Q^t K_j^T (128 x 128, fp32 in TMEM) for both tiles,
//               each as soon as softmax t has read the previous one;
//   warps 2, 3  issue O^t += P^t V_j for tile 0 and tile 1 (128 x 64,
//               accumulated in TMEM, P read from TMEM).  One thread issues a
//               tcgen05.mma only about every 120 cycles whatever its shape, and
//               an N = 64 MMA is 32 cycles of work, so the P V MMAs of each tile
//               get their own issuing thread;
//   warps 4-7   softmax of tile 0, warps 8-11 softmax of tile 1: one query row
//               per thread.  Each reads its S row from TMEM with the row
//               maximum computed by the load itself (tcgen05.ld.red, sm_103a),
//               updates the running max and sum, computes P = 2^(s*c - m*c) as bf16 pairs
//               in registers and, once the previous P V has read the tile's P
//               columns, writes them to tensor memory, where the P V MMA reads
//               its A operand.
// setmaxnreg moves registers from the load / MMA warpgroup (56 per thread) to
// the softmax warpgroups (224), which hold a whole S row and P row at once.
// The running max is only raised when it grows by more than 2^8 (in the exp2
// domain); then the thread rescales its O row in TMEM first.  P, O and the sum
// always use the same max, so the result is exact up to rounding.
#include <cudaTypedefs.h>

#include "common.cuh"
#include "kernels.h"
#include "tc_ptx.cuh"

namespace sr {
namespace {

using namespace tc;

constexpr int kDh = 64;
constexpr int kQTile = 128, kQTiles = 2, kBQ = kQTile * kQTiles;
constexpr int kKV = 128;
constexpr int kStages = 3;                                    // K ring and V ring
constexpr int kThreads = 384;
constexpr int kTileBytes = kQTile * kDh * 2;                  // 16 KB: 128 rows x 128 B
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColS = 0;      // S^t at columns [128 t, 128 t + 128)
constexpr uint32_t kColO = 256;    // O^t at columns [256 + 64 t, 256 + 64 t + 64)
constexpr uint32_t kColP = 384;    // P^t (bf16 pairs) at columns [384 + 64 t, 384 + 64 t + 64)
// raise the running max only when it grows by more than 8 in the exp2 domain
constexpr float kRescaleLog2 = 8.0f;

struct AttSmem {
  uint64_t q_full, q_free;
  uint64_t k_full[kStages], k_empty[kStages], v_full[kStages], v_empty[kStages];
  uint64_t s_full[kQTiles], s_free[kQTiles], p_full[kQTiles], pv_done[kQTiles];
  uint64_t drain[1 + kQTiles];      // the S issuer, then each P V issuer
  uint32_t tmem_base;
  int abort;
};

constexpr size_t kSmemBytes = 1024 /*align*/ + size_t(kQTiles) * kTileBytes +
                              size_t(kStages) * 2 * kTileBytes + 256;
static_assert(sizeof(AttSmem) <= 256, "barrier block outgrew its reserve");

// 32x32b.x128 TMEM load: a thread's 128 consecutive columns of its lane (as
// four tmem_ld32 would load them) and, per thread, the maximum of those 128
// values (sm_103a: tcgen05.ld.red)
__device__ __forceinline__ void tmem_ld128_max(uint32_t taddr, uint32_t (&r)[128], float& m) {
  asm volatile(
      "tcgen05.ld.red.sync.aligned.32x32b.x128.max.f32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32, %33, %34, %35, %36, %37, %38, %39, %40, %41, %42, %43, %44, %45, %46, %47, %48, %49, %50, %51, %52, %53, %54, %55, %56, %57, %58, %59, %60, %61, %62, %63, %64, %65, %66, %67, %68, %69, %70, %71, %72, %73, %74, %75, %76, %77, %78, %79, %80, %81, %82, %83, %84, %85, %86, %87, %88, %89, %90, %91, %92, %93, %94, %95, %96, %97, %98, %99, %100, %101, %102, %103, %104, %105, %106, %107, %108, %109, %110, %111, %112, %113, %114, %115, %116, %117, %118, %119, %120, %121, %122, %123, %124, %125, %126, %127}, %128, [%129];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
        "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]),
        "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]),
        "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
        "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63]),
        "=r"(r[64]), "=r"(r[65]), "=r"(r[66]), "=r"(r[67]), "=r"(r[68]), "=r"(r[69]), "=r"(r[70]), "=r"(r[71]),
        "=r"(r[72]), "=r"(r[73]), "=r"(r[74]), "=r"(r[75]), "=r"(r[76]), "=r"(r[77]), "=r"(r[78]), "=r"(r[79]),
        "=r"(r[80]), "=r"(r[81]), "=r"(r[82]), "=r"(r[83]), "=r"(r[84]), "=r"(r[85]), "=r"(r[86]), "=r"(r[87]),
        "=r"(r[88]), "=r"(r[89]), "=r"(r[90]), "=r"(r[91]), "=r"(r[92]), "=r"(r[93]), "=r"(r[94]), "=r"(r[95]),
        "=r"(r[96]), "=r"(r[97]), "=r"(r[98]), "=r"(r[99]), "=r"(r[100]), "=r"(r[101]), "=r"(r[102]), "=r"(r[103]),
        "=r"(r[104]), "=r"(r[105]), "=r"(r[106]), "=r"(r[107]), "=r"(r[108]), "=r"(r[109]), "=r"(r[110]), "=r"(r[111]),
        "=r"(r[112]), "=r"(r[113]), "=r"(r[114]), "=r"(r[115]), "=r"(r[116]), "=r"(r[117]), "=r"(r[118]), "=r"(r[119]),
        "=r"(r[120]), "=r"(r[121]), "=r"(r[122]), "=r"(r[123]), "=r"(r[124]), "=r"(r[125]), "=r"(r[126]), "=r"(r[127]),
        "=f"(m)
      : "r"(taddr));
}

// kPersist: a CTA takes the work items (one (sample, head, 256-query block)
// each) blockIdx.x, blockIdx.x + gridDim.x, ... in turn, with its barriers,
// tensor memory and K/V rings kept across items; the next item's Q is loaded
// once the previous item's S MMAs have read Q, and its first P V overwrites O
// only after the previous item's epilogue has read O (the softmax threads read
// O before they signal the next item's first P).  Without kPersist every CTA
// has one item (the grid is the item count).
template <bool kPersist>
__global__ void __launch_bounds__(kThreads, 1)
attention_tc_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmKV,
                    bf16* __restrict__ out, int Tq, int Tkv, int heads, int qcol0, int kcol0,
                    int vcol0, int items, unsigned int* fault) {
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* base = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* sQ = base;                                  // 2 x 16 KB
  unsigned char* sK = sQ + kQTiles * kTileBytes;             // stages x 16 KB
  unsigned char* sV = sK + kStages * kTileBytes;             // stages x 16 KB
  AttSmem* sm = reinterpret_cast<AttSmem*>(sV + kStages * kTileBytes);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int qblocks = (Tq + kBQ - 1) / kBQ;
  const int D = heads * kDh;
  const int nkv = (Tkv + kKV - 1) / kKV;
  const int item_step = kPersist ? int(gridDim.x) : items;

  if (threadIdx.x == 0) {
    mbar_init(&sm->q_full, 1);
    mbar_init(&sm->q_free, 1);
    for (int s = 0; s < kStages; ++s) {
      // a K stage is released by the S issuer, a V stage by both P V issuers
      mbar_init(&sm->k_full[s], 1); mbar_init(&sm->k_empty[s], 1);
      mbar_init(&sm->v_full[s], 1); mbar_init(&sm->v_empty[s], kQTiles);
    }
    for (int t = 0; t < kQTiles; ++t) {
      mbar_init(&sm->s_full[t], 1);
      mbar_init(&sm->s_free[t], kQTile);
      mbar_init(&sm->p_full[t], kQTile);
      mbar_init(&sm->pv_done[t], 1);
    }
    for (int d = 0; d < 1 + kQTiles; ++d) mbar_init(&sm->drain[d], 1);
    sm->abort = 0;
    fence_mbar_init();
  }
  if (warp == 0 && lane == 0) {
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmKV);
  }
  if (warp == 1) tmem_alloc(&sm->tmem_base, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm->tmem_base;
  volatile int* abort = &sm->abort;
  pdl_wait();      // the previous kernel's writes are visible from here
  pdl_trigger();

  if (warp < 4) {
    // registers: 56 per thread for the load / MMA warpgroup, 224 for the two
    // softmax warpgroups; 128 * 56 + 256 * 224 = 384 * 168, the launch's total
    // (the launcher checks that the kernel was built with 168)
    asm volatile("setmaxnreg.dec.sync.aligned.u32 56;\n" ::: "memory");
    if (warp == 0) {
      // ------------------------------------------------------------- TMA loads
      // per item: the two Q tiles, then K_j and V_j into their rings
      if (lane == 0) {
        // stages holding a load, and the parity of the phase each last used
        uint32_t kissued = 0, vissued = 0, kpar = 0, vpar = 0;
        int st = 0, q_loads = 0;
        uint32_t ph = 0;
        bool ok = true;
        for (int item = blockIdx.x, it = 0; ok && item < items; item += item_step, ++it) {
          const int bh = item / qblocks, qb = item % qblocks;
          const int b = bh / heads, h = bh % heads;
          // a persistent CTA reloads Q once the previous item's S MMAs have read it
          if (kPersist && it > 0 && !(ok = mbar_wait(&sm->q_free, (it - 1) & 1, abort, fault))) break;
          mbar_arrive_expect_tx(&sm->q_full, kQTiles * kTileBytes);
          for (int t = 0; t < kQTiles; ++t)
            tma_load_3d(&tmQ, sQ + t * kTileBytes, &sm->q_full, qcol0 + h * kDh,
                        qb * kBQ + t * kQTile, b);
          ++q_loads;
          const int kcol = kcol0 + h * kDh, vcol = vcol0 + h * kDh;
          for (int j = 0; j < nkv; ++j) {
            // a K stage frees once both tiles' S MMAs of key tile j - kStages are done
            if (!(ok = mbar_wait(&sm->k_empty[st], ph ^ 1, abort, fault))) break;
            mbar_arrive_expect_tx(&sm->k_full[st], kTileBytes);
            tma_load_3d(&tmKV, sK + st * kTileBytes, &sm->k_full[st], kcol, j * kKV, b);
            kissued |= 1u << st;
            kpar = (kpar & ~(1u << st)) | (ph << st);
            // a V stage once both tiles' P V MMAs of that key tile are
            if (!(ok = mbar_wait(&sm->v_empty[st], ph ^ 1, abort, fault))) break;
            mbar_arrive_expect_tx(&sm->v_full[st], kTileBytes);
            tma_load_3d(&tmKV, sV + st * kTileBytes, &sm->v_full[st], vcol, j * kKV, b);
            vissued |= 1u << st;
            vpar = (vpar & ~(1u << st)) | (ph << st);
            if (++st == kStages) { st = 0; ph ^= 1; }
          }
          if constexpr (!kPersist) break;
        }
        // every issued load lands before the CTA may exit
        int no_abort = 0;
        if (q_loads > 0) mbar_wait(&sm->q_full, uint32_t(q_loads - 1) & 1u, &no_abort, fault);
        for (int s = 0; s < kStages; ++s) {
          if (kissued & (1u << s)) mbar_wait(&sm->k_full[s], (kpar >> s) & 1u, &no_abort, fault);
          if (vissued & (1u << s)) mbar_wait(&sm->v_full[s], (vpar >> s) & 1u, &no_abort, fault);
        }
      }
    } else if (warp == 1) {
      // ------------------------------------------------------------- S MMAs
      // S^t = Q^t K_j^T for both tiles, each once softmax t has read S^t of the
      // previous key tile (of this item or, persistent, of the previous item)
      if (lane == 0) {
        constexpr uint32_t idesc_s = idesc_bf16(kQTile, kKV);                 // K-major A, B
        int st = 0, g = 0;                 // g: key tiles of earlier items
        uint32_t ph = 0;
        bool ok = true;
        for (int item = blockIdx.x, it = 0; ok && item < items; item += item_step, ++it) {
          const int gb = kPersist ? g : 0;
          if (!(ok = mbar_wait(&sm->q_full, uint32_t(it) & 1u, abort, fault))) break;
          for (int j = 0; j < nkv && ok; ++j) {
            if (!(ok = mbar_wait(&sm->k_full[st], ph, abort, fault))) break;
            const uint32_t ka = smem_u32(sK + st * kTileBytes);
            for (int t = 0; t < kQTiles && ok; ++t) {
              if (gb + j > 0 && !(ok = mbar_wait(&sm->s_free[t], (gb + j - 1) & 1, abort, fault))) break;
              tc_fence_after();
              const uint32_t qa = smem_u32(sQ + t * kTileBytes);
              const uint32_t dS = tmem + kColS + uint32_t(t * kKV);
#pragma unroll
              for (int k = 0; k < kDh / 16; ++k)
                mma_bf16(dS, sw128_desc(qa + 32 * k), sw128_desc(ka + 32 * k), idesc_s,
                         k > 0 ? 1u : 0u);
              mma_commit(&sm->s_full[t]);
            }
            if (!ok) break;
            mma_commit(&sm->k_empty[st]);
            if (++st == kStages) { st = 0; ph ^= 1; }
          }
          if (!ok) break;
          // Q may be reloaded once this item's S MMAs are done
          if constexpr (kPersist) mma_commit(&sm->q_free);
          g += nkv;
          if constexpr (!kPersist) break;
        }
        int no_abort = 0;
        mma_commit(&sm->drain[0]);
        mbar_wait(&sm->drain[0], 0, &no_abort, fault);
      }
    } else {
      // ------------------------------------------------------------- P V MMAs
      // warp 2 for tile 0, warp 3 for tile 1: O^t += P^t_j V_j (128 x 64,
      // accumulated in TMEM), P read from TMEM (64 columns of bf16 pairs).  An
      // item's first P V overwrites O; its P is signalled only after the
      // softmax threads have read the previous item's O.
      if (lane == 0) {
        const int t = warp - 2;
        constexpr uint32_t idesc_o = idesc_bf16(kQTile, kDh, false, true);   // V is MN-major
        const uint32_t dO = tmem + kColO + uint32_t(t * kDh);
        const uint32_t aP = tmem + kColP + uint32_t(t * (kKV / 2));
        bool ok = true;
        int st = 0, g = 0;
        uint32_t ph = 0;
        for (int item = blockIdx.x; ok && item < items; item += item_step) {
          const int gb = kPersist ? g : 0;
          for (int j = 0; j < nkv && ok; ++j) {
            if (!(ok = mbar_wait(&sm->v_full[st], ph, abort, fault))) break;
            if (!(ok = mbar_wait(&sm->p_full[t], (gb + j) & 1, abort, fault))) break;
            tc_fence_after();
            const uint32_t va = smem_u32(sV + st * kTileBytes);
#pragma unroll
            for (int k = 0; k < kKV / 16; ++k)
              mma_bf16_ts(dO, aP + uint32_t(k * 8), sw128_desc_mn(va + k * 2048), idesc_o,
                          (j | k) != 0 ? 1u : 0u);
            mma_commit(&sm->pv_done[t]);
            mma_commit(&sm->v_empty[st]);
            if (++st == kStages) { st = 0; ph ^= 1; }
          }
          g += nkv;
          if constexpr (!kPersist) break;
        }
        int no_abort = 0;
        mma_commit(&sm->drain[1 + t]);
        mbar_wait(&sm->drain[1 + t], 0, &no_abort, fault);
      }
    }
  } else {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 224;\n" ::: "memory");
    // ------------------------------------------------------------- softmax
    const int t = (warp - 4) >> 2;                 // query tile of this warpgroup
    const int quarter = warp & 3;                  // TMEM lane quarter
    const int r = quarter * 32 + lane;             // row within the tile
    const uint32_t lane_off = uint32_t(quarter * 32) << 16;
    const uint32_t tS = tmem + lane_off + kColS + uint32_t(t * kKV);
    const uint32_t tO = tmem + lane_off + kColO + uint32_t(t * kDh);
    const uint32_t tP = tmem + lane_off + kColP + uint32_t(t * (kKV / 2));
    const float c = 0.125f * 1.4426950408889634f;  // 1/sqrt(64) * log2(e)
    const float thresh = kRescaleLog2 / c;         // the same threshold in score units
    const uint64_t c2 = pk2(c, c);
    bool ok = true;
    int g = 0;                                     // key tiles of earlier items
    for (int item = blockIdx.x; ok && item < items; item += item_step) {
    const int gb = kPersist ? g : 0;
    const int bh = item / qblocks, qb = item % qblocks;
    const int b = bh / heads, h = bh % heads;
    const int q0 = qb * kBQ;
    float m_run = -INFINITY, l_run = 0.f;
    for (int j = 0; j < nkv; ++j) {
      ok = __all_sync(0xffffffffu, mbar_wait(&sm->s_full[t], (gb + j) & 1, abort, fault));
      if (!ok) break;
      tc_fence_after();
      // S with its row maximum: one load of the row's 128 columns, which also
      // reduces them to their maximum
      static_assert(kKV == 128, "one 128-column load per S row");
      uint32_t s[kKV / 32][32];
      float tmax;
      tmem_ld128_max(tS, reinterpret_cast<uint32_t (&)[kKV]>(s), tmax);
      tmem_wait_ld();
      tc_fence_before();
      mbar_arrive(&sm->s_free[t]);                 // S may now be overwritten
      const int valid = Tkv - j * kKV;             // keys of this tile that exist
      if (valid < kKV) {
        // keys past the end are zero-filled (S = 0 there): mask them and take
        // the maximum over the keys that exist
        tmax = -INFINITY;
#pragma unroll
        for (int i = 0; i < kKV; ++i) {
          if (i >= valid) s[i / 32][i % 32] = __float_as_uint(-INFINITY);
          tmax = fmaxf(tmax, __uint_as_float(s[i / 32][i % 32]));
        }
      }
      float alpha = 1.f;
      bool rescale = false;
      if (j == 0) {
        m_run = tmax;
      } else if (tmax > m_run + thresh) {
        alpha = ex2((m_run - tmax) * c);
        m_run = tmax;
        l_run *= alpha;
        rescale = true;
      }
      // P = 2^(s c - m c) as bf16 pairs, held in registers until the previous
      // P V has released the tile's P columns: key 2i and 2i+1 of this row share
      // column i of the tile's P region (the A operand of P V)
      const float mc = m_run * c;
      const uint64_t nmc2 = pk2(-mc, -mc);
      uint64_t ls2[2] = {pk2(0.f, 0.f), pk2(0.f, 0.f)};
      uint32_t w[kKV / 64][32];
#pragma unroll
      for (int cc = 0; cc < kKV / 32; ++cc) {
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          const int i0 = 32 * cc + 2 * q;
          const uint64_t arg = fma2(pk2(__uint_as_float(s[i0 / 32][i0 % 32]),
                                        __uint_as_float(s[(i0 + 1) / 32][(i0 + 1) % 32])),
                                    c2, nmc2);
          float a0, a1;
          up2(arg, a0, a1);
          const uint64_t p2 = pk2(ex2(a0), ex2(a1));
          ls2[q & 1] = add2(ls2[q & 1], p2);
          float p0, p1;
          up2(p2, p0, p1);
          w[cc / 2][(cc % 2) * 16 + q] = pack_bf16x2(p0, p1);
        }
      }
      {
        float l0, l1, l2, l3;
        up2(ls2[0], l0, l1);
        up2(ls2[1], l2, l3);
        l_run += (l0 + l1) + (l2 + l3);
      }
      // P and O of this tile are free once the previous P V has completed
      if (gb + j >= 1) {
        ok = __all_sync(0xffffffffu, mbar_wait(&sm->pv_done[t], (gb + j - 1) & 1, abort, fault));
        if (!ok) break;
        tc_fence_after();
      }
#pragma unroll
      for (int hh = 0; hh < kKV / 64; ++hh) tmem_st32(tP + uint32_t(hh * 32), w[hh]);
      // a raised max rescales O, which holds every earlier P V product
      if (__any_sync(0xffffffffu, rescale)) {
        uint32_t o[32];
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          tmem_ld32(tO + uint32_t(half * 32), o);
          tmem_wait_ld();
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * alpha);
          tmem_st32(tO + uint32_t(half * 32), o);
        }
      }
      tmem_wait_st();
      tc_fence_before();
      mbar_arrive(&sm->p_full[t]);
    }
    // epilogue: O / l for the rows that exist (the last P V implies all earlier ones)
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&sm->pv_done[t], (gb + nkv - 1) & 1, abort, fault));
    if (ok) {
      tc_fence_after();
      uint32_t o[2][32];
      tmem_ld32(tO, o[0]);
      tmem_ld32(tO + 32, o[1]);
      tmem_wait_ld();
      const int row = q0 + t * kQTile + r;
      if (row < Tq) {
        const float inv = 1.f / l_run;
        uint4* dst = reinterpret_cast<uint4*>(out + (size_t(b) * Tq + row) * D + h * kDh);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const uint32_t* q = &o[i / 4][(i % 4) * 8];
          dst[i] = make_uint4(pack_bf16x2(__uint_as_float(q[0]) * inv, __uint_as_float(q[1]) * inv),
                              pack_bf16x2(__uint_as_float(q[2]) * inv, __uint_as_float(q[3]) * inv),
                              pack_bf16x2(__uint_as_float(q[4]) * inv, __uint_as_float(q[5]) * inv),
                              pack_bf16x2(__uint_as_float(q[6]) * inv, __uint_as_float(q[7]) * inv));
        }
      }
    }
    g += nkv;
    if constexpr (!kPersist) break;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

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


// 3-D bf16 tensor map over [B, T, C] (row-major), box 64 columns x 128 rows x 1
cudaError_t make_map_btc(CUtensorMap* map, const void* ptr, int B, int T, uint64_t C) {
  cudaError_t e = get_encoder();
  if (e != cudaSuccess) return e;
  cuuint64_t dims[3] = {C, uint64_t(T), uint64_t(B)};
  cuuint64_t strides[2] = {C * 2, C * 2 * uint64_t(T)};
  cuuint32_t box[3] = {kDh, kKV, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  CUresult r = g_encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS ? cudaSuccess : cudaErrorInvalidValue;
}

// Sets the kernel's attributes once and returns how many of its CTAs fit on the
// GPU at once (one per SM: the CTA takes all 512 tensor-memory columns).
template <bool kPersist>
cudaError_t prepare(int* resident) {
  static int cache[kMaxDevices] = {};
  const int slot = device_slot();
  if (slot < 0) return cudaErrorInvalidDevice;
  int& cached = cache[slot];
  if (cached == 0) {
    cudaFuncAttributes fa;
    cudaError_t e = cudaFuncGetAttributes(&fa, attention_tc_kernel<kPersist>);
    if (e != cudaSuccess) return e;
    if (fa.numRegs < 168) return cudaErrorInvalidConfiguration;   // the register split needs 168
    e = cudaFuncSetAttribute(attention_tc_kernel<kPersist>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize, int(kSmemBytes));
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0, per_sm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, attention_tc_kernel<kPersist>,
                                                      kThreads, kSmemBytes);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    cached = sms * per_sm;
  }
  *resident = cached;
  return cudaSuccess;
}

// Short key sequences (at most kPersistMaxKeyTiles key tiles) run on a
// persistent grid of one CTA per SM: there a CTA's fixed cost (barrier setup,
// tensor-memory allocation, the first loads, the epilogue and teardown, about
// 3.3 us) is a large part of an item's work.  Longer ones run one CTA per item,
// where the persistent loop's extra state costs more than it saves.
constexpr int kPersistMaxKeyTiles = 16;

cudaError_t launch(const CUtensorMap& tq, const CUtensorMap& tkv, void* out, int B, int Tq,
                   int Tkv, int heads, int qcol0, int kcol0, int vcol0, unsigned int* fault,
                   cudaStream_t s) {
  const int items = B * heads * ((Tq + kBQ - 1) / kBQ);
  const int nkv = (Tkv + kKV - 1) / kKV;
  int resident = 0;
  if (nkv <= kPersistMaxKeyTiles) {
    cudaError_t e = prepare<true>(&resident);
    if (e != cudaSuccess) return e;
    if (items > resident)
      return launch_k(attention_tc_kernel<true>, dim3(resident), dim3(kThreads), kSmemBytes, s, 1,
                      tq, tkv, static_cast<bf16*>(out), Tq, Tkv, heads, qcol0, kcol0, vcol0, items,
                      fault);
  }
  cudaError_t e = prepare<false>(&resident);
  if (e != cudaSuccess) return e;
  return launch_k(attention_tc_kernel<false>, dim3(items), dim3(kThreads), kSmemBytes, s, 1, tq, tkv,
                  static_cast<bf16*>(out), Tq, Tkv, heads, qcol0, kcol0, vcol0, items, fault);
}

}  // namespace

cudaError_t launch_attention_tc(const void* qkv, void* out, int B, int T, int heads,
                                unsigned int* fault, cudaStream_t s) {
  const int D = heads * kDh;
  CUtensorMap tm;
  cudaError_t e = make_map_btc(&tm, qkv, B, T, uint64_t(3) * D);   // [B, T, 3D]: q | k | v
  if (e != cudaSuccess) return e;
  return launch(tm, tm, out, B, T, T, heads, 0, D, 2 * D, fault, s);
}

cudaError_t launch_cross_attention_tc(const void* q, const void* kv, void* out, int B, int Tq,
                                      int Tkv, int heads, unsigned int* fault, cudaStream_t s) {
  const int D = heads * kDh;
  CUtensorMap tq, tkv;
  cudaError_t e = make_map_btc(&tq, q, B, Tq, uint64_t(D));        // [B, Tq, D]
  if (e != cudaSuccess) return e;
  e = make_map_btc(&tkv, kv, B, Tkv, uint64_t(2) * D);             // [B, Tkv, 2D]: k | v
  if (e != cudaSuccess) return e;
  return launch(tq, tkv, out, B, Tq, Tkv, heads, 0, 0, D, fault, s);
}

}  // namespace sr
