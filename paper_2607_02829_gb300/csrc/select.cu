// Token selection (Sec. 3.2 random selection; App. B.2 activation-norm and
// gradient (Laplacian) selectors).
//
// All selectors reduce to one primitive: per sample, keep the K smallest keys
// (ties broken by the lower token index) and emit their token indices in
// ascending order.  One CTA owns one sample: its L keys sit in shared memory, a
// most-significant-digit radix select (8-bit digits, stopping once the K-th
// smallest key's digit bin is kept whole) finds the threshold and how many keys
// equal to it must be kept, and an ordered block-wide compaction writes the
// selected indices, which come out sorted by construction.  Work per sample is O(L * passes); HBM traffic is the index
// write (4 B per selected token) plus, for the score-based selectors, the
// scores: one pass over x computes them (the L2 norms, or the Laplacian on the
// patch grid), unless the forward's FC2 epilogue already has the norms.
#include "common.cuh"
#include "kernels.h"

namespace sr {
namespace {

constexpr int kSelThreads = 1024;
constexpr int kSelMaxL = 24576;   // 192 KB of 8-byte keys in shared memory

// SplitMix64 output function (Steele, Lea & Flood, OOPSLA 2014).
__device__ __forceinline__ uint64_t splitmix64_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// Scores in descending order become keys in ascending order (equal scores give
// equal keys, so ties fall to the index order of the compaction).
__device__ __forceinline__ uint32_t desc_key(float score) {
  uint32_t u = __float_as_uint(score);
  uint32_t asc = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ~asc;
}

// Block-wide exclusive prefix sum of `v` in thread order; returns the thread's
// exclusive prefix and writes the block total to *total.
__device__ __forceinline__ int block_excl_sum(int v, int* warp_tot, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int t = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += t;
  }
  if (lane == 31) warp_tot[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const int nw = blockDim.x >> 5;
    const int w = lane < nw ? warp_tot[lane] : 0;
    int wi = w;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int t = __shfl_up_sync(0xffffffffu, wi, o);
      if (lane >= o) wi += t;
    }
    if (lane < nw) warp_tot[lane] = wi - w;      // exclusive warp offsets
    if (lane == 31) *total = wi;
  }
  __syncthreads();
  const int r = warp_tot[warp] + incl - v;
  __syncthreads();   // warp_tot is reused by the next call
  return r;
}

// Writes, in ascending order, the indices of the K smallest of the L keys
// (ties to the lower index).  A most-significant-digit radix select (8-bit
// digits) narrows a prefix of the K-th smallest key; it stops as soon as every
// key under the current prefix is kept, which for random keys happens after a
// few digits.  The compaction then gives each thread a contiguous range of
// indices: two block scans (of the kept keys equal to the threshold, then of
// all kept keys) place every index.
template <typename Key>
__device__ void select_smallest_sorted(const Key* keys, int L, int K, int32_t* out_idx) {
  __shared__ int hist[256];
  __shared__ int warp_tot[32];
  __shared__ int s_total;
  __shared__ Key s_prefix;
  __shared__ int s_krem;
  __shared__ int s_whole;      // every key under the prefix is kept
  const int tid = threadIdx.x;
  if (tid == 0) { s_prefix = 0; s_krem = K; s_whole = 0; }
  Key mask = 0;
  __syncthreads();
  // ---- radix select of the K-th smallest key, most significant digit first
  for (int shift = int(sizeof(Key) * 8) - 8; shift >= 0; shift -= 8) {
    for (int i = tid; i < 256; i += blockDim.x) hist[i] = 0;
    __syncthreads();
    const Key prefix = s_prefix;
    for (int i = tid; i < L; i += blockDim.x) {
      const Key k = keys[i];
      if ((k & mask) == prefix) atomicAdd(&hist[int((k >> shift) & 0xff)], 1);
    }
    __syncthreads();
    if (tid < 32) {
      // lane l owns bins 8l .. 8l+7
      int c[8], s = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) { c[j] = hist[8 * tid + j]; s += c[j]; }
      int incl = s;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        int t = __shfl_up_sync(0xffffffffu, incl, o);
        if (tid >= o) incl += t;
      }
      const int krem = s_krem;
      const int excl = incl - s;
      if (excl < krem && krem <= incl) {
        int acc = excl, d = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (acc + c[j] >= krem) { d = j; break; }
          acc += c[j];
        }
        s_prefix = prefix | (Key(8 * tid + d) << shift);
        s_krem = krem - acc;
        s_whole = c[d] == krem - acc;
      }
    }
    mask |= Key(0xff) << shift;
    __syncthreads();
    if (s_whole) break;
  }
  // keys are compared under `mask`: below the threshold T they are kept; equal
  // to it, the first keep_eq of them (all of them when the select stopped early)
  const Key T = s_prefix;
  const int keep_eq = s_krem;
  // ---- compaction over contiguous ranges of indices, one range per thread; an
  // odd range length keeps a warp's reads of its 32 ranges on distinct banks
  const int per = ((L + int(blockDim.x) - 1) / int(blockDim.x)) | 1;
  const int i0 = min(L, tid * per), i1 = min(L, i0 + per);
  int n_eq = 0;
  for (int i = i0; i < i1; ++i) n_eq += (keys[i] & mask) == T;
  int eq_rank = block_excl_sum(n_eq, warp_tot, &s_total);
  int n_keep = 0;
  for (int i = i0, r = eq_rank; i < i1; ++i) {
    const Key km = keys[i] & mask;
    if (km < T) ++n_keep;
    else if (km == T) n_keep += r++ < keep_eq;
  }
  int pos = block_excl_sum(n_keep, warp_tot, &s_total);
  for (int i = i0; i < i1; ++i) {
    const Key km = keys[i] & mask;
    bool keep = km < T;
    if (km == T) keep = eq_rank++ < keep_eq;
    if (keep) out_idx[pos++] = i;
  }
}

__global__ void __launch_bounds__(kSelThreads)
select_random_kernel(int L, int K, uint64_t seed, int shared, int32_t* idx) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  pdl_wait();      // the previous kernel's writes are visible from here
  pdl_trigger();

  uint64_t* keys = reinterpret_cast<uint64_t*>(smem_raw);
  const int b = blockIdx.x;
  const uint64_t bb = shared ? 0ull : uint64_t(b);
  for (int i = threadIdx.x; i < L; i += blockDim.x) {
    const uint64_t ctr = 1ull + bb * uint64_t(L) + uint64_t(i);
    keys[i] = splitmix64_mix(seed + 0x9E3779B97F4A7C15ull * ctr);
  }
  __syncthreads();
  select_smallest_sorted<uint64_t>(keys, L, K, idx + size_t(b) * K);
}

__global__ void __launch_bounds__(kSelThreads)
select_topk_kernel(int L, int K, const float* __restrict__ score, int parts, int32_t* idx) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  pdl_wait();      // the previous kernel's writes are visible from here
  pdl_trigger();

  uint32_t* keys = reinterpret_cast<uint32_t*>(smem_raw);
  const int b = blockIdx.x;
  // a token's score is the sum of its `parts` partial sums, added in slot order
  for (int i = threadIdx.x; i < L; i += blockDim.x) {
    const float* sp = score + (size_t(b) * L + i) * parts;
    float v = sp[0];
    for (int p = 1; p < parts; ++p) v += sp[p];
    keys[i] = desc_key(v);
  }
  __syncthreads();
  select_smallest_sorted<uint32_t>(keys, L, K, idx + size_t(b) * K);
}

// One warp per token: every fp32 stream value is rounded to the storage dtype T
// (the activation as the model stores it), then squared and summed in fp32.
template <typename T>
__global__ void __launch_bounds__(256)
token_sq_norms_kernel(const float* __restrict__ x, int rows, int D, float* __restrict__ score) {
  pdl_wait();      // the previous kernel's writes are visible from here
  pdl_trigger();
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= rows) return;
  const float4* row = reinterpret_cast<const float4*>(x + size_t(warp) * D);
  const int nv = D / 4;
  float acc = 0.f;
  for (int v = lane; v < nv; v += 32) {
    const float4 q = __ldg(row + v);
    const float f[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float r = Elem<T>::to_f(Elem<T>::from_f(f[j]));
      acc = fmaf(r, r, acc);
    }
  }
  acc = warp_sum(acc);
  if (lane == 0) score[warp] = acc;
}

// One warp per token (i, j) of the patch grid: the 5-point Laplacian of its row
// of the stream, x(i-1,j) + x(i+1,j) + x(i,j-1) + x(i,j+1) - 4 x(i,j), with
// longitude periodic and the first and last latitude rows reflected onto
// themselves; every value rounded to the storage dtype T first, the squared
// norm of the stencil accumulated in fp32.  Each row is read by five warps, so
// the neighbours' reads come from L2.
template <typename T>
__global__ void __launch_bounds__(256)
token_laplacian_kernel(const float* __restrict__ x, int B, int L, int W, int D,
                       float* __restrict__ score) {
  pdl_wait();      // the previous kernel's writes are visible from here
  pdl_trigger();
  const int t = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (t >= B * L) return;
  const int b = t / L, tok = t % L;
  const int H = L / W, i = tok / W, j = tok % W;
  const size_t base = size_t(b) * L;
  const float4* c = reinterpret_cast<const float4*>(x + (base + tok) * D);
  const float4* n = reinterpret_cast<const float4*>(x + (base + size_t(i > 0 ? i - 1 : 0) * W + j) * D);
  const float4* so = reinterpret_cast<const float4*>(
      x + (base + size_t(i + 1 < H ? i + 1 : H - 1) * W + j) * D);
  const float4* w = reinterpret_cast<const float4*>(x + (base + size_t(i) * W + (j + W - 1) % W) * D);
  const float4* e = reinterpret_cast<const float4*>(x + (base + size_t(i) * W + (j + 1) % W) * D);
  auto rd = [](float v) { return Elem<T>::to_f(Elem<T>::from_f(v)); };
  float acc = 0.f;
  for (int v = lane; v < D / 4; v += 32) {
    const float4 qc = __ldg(c + v), qn = __ldg(n + v), qs = __ldg(so + v), qw = __ldg(w + v),
                 qe = __ldg(e + v);
    const float fc[4] = {qc.x, qc.y, qc.z, qc.w}, fn[4] = {qn.x, qn.y, qn.z, qn.w},
                fs[4] = {qs.x, qs.y, qs.z, qs.w}, fw[4] = {qw.x, qw.y, qw.z, qw.w},
                fe[4] = {qe.x, qe.y, qe.z, qe.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float lap = ((rd(fn[k]) + rd(fs[k])) + (rd(fw[k]) + rd(fe[k]))) - 4.0f * rd(fc[k]);
      acc = fmaf(lap, lap, acc);
    }
  }
  acc = warp_sum(acc);
  if (lane == 0) score[t] = acc;
}

}  // namespace

int select_max_L() { return kSelMaxL; }

cudaError_t launch_token_laplacian(DType dt, const float* x, int B, int L, int grid_w, int D,
                                   float* score, cudaStream_t s) {
  if (grid_w < 1 || L % grid_w != 0 || D % 4 != 0) return cudaErrorInvalidValue;
  const int blocks = (B * L + 7) / 8;
  if (dt == DType::BF16)
    return launch_k(token_laplacian_kernel<bf16>, dim3(blocks), dim3(256), 0, s, 1, x, B, L, grid_w,
                    D, score);
  return launch_k(token_laplacian_kernel<float>, dim3(blocks), dim3(256), 0, s, 1, x, B, L, grid_w, D,
                  score);
}

// Raises a kernel's dynamic shared-memory limit only when a launch needs more
// than an earlier one set (so that calls after the first, which may be inside a
// stream capture, make no attribute change).
template <typename Kernel>
static cudaError_t ensure_smem(Kernel kernel, size_t smem, int* current) {
  if (int(smem) <= *current) return cudaSuccess;
  const cudaError_t e =
      cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e == cudaSuccess) *current = int(smem);
  return e;
}
static int g_random_smem[kMaxDevices] = {}, g_topk_smem[kMaxDevices] = {};

cudaError_t launch_select_random(int B, int L, int K, uint64_t seed, int shared, int32_t* idx,
                                 cudaStream_t s) {
  const size_t smem = size_t(L) * sizeof(uint64_t);
  const int dev = device_slot();
  if (dev < 0) return cudaErrorInvalidDevice;
  cudaError_t e = ensure_smem(select_random_kernel, smem, &g_random_smem[dev]);
  if (e != cudaSuccess) return e;
  return launch_k(select_random_kernel, dim3(B), dim3(kSelThreads), smem, s, 1, L, K, seed, shared,
                  idx);
}

cudaError_t launch_select_topk(int B, int L, int K, const float* score, int32_t* idx,
                               cudaStream_t s, int parts) {
  const size_t smem = size_t(L) * sizeof(uint32_t);
  const int dev = device_slot();
  if (dev < 0) return cudaErrorInvalidDevice;
  cudaError_t e = ensure_smem(select_topk_kernel, smem, &g_topk_smem[dev]);
  if (e != cudaSuccess) return e;
  return launch_k(select_topk_kernel, dim3(B), dim3(kSelThreads), smem, s, 1, L, K, score, parts, idx);
}

cudaError_t launch_token_sq_norms(DType dt, const float* x, int rows, int D, float* score,
                                  cudaStream_t s) {
  const int blocks = (rows + 7) / 8;
  if (dt == DType::BF16)
    return launch_k(token_sq_norms_kernel<bf16>, dim3(blocks), dim3(256), 0, s, 1, x, rows, D, score);
  return launch_k(token_sq_norms_kernel<float>, dim3(blocks), dim3(256), 0, s, 1, x, rows, D, score);
}

}  // namespace sr
