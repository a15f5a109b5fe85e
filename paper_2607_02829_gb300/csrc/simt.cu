// CUDA-core (FFMA) kernels for the fp32 configuration: the block GEMMs with
// their fused epilogues and the attention core.  fp32 end to end, because TF32
// tensor cores would not hold the fp32 tolerance.  These kernels serve the
// small fp32 model (D = 256); the bf16 path runs on the tcgen05 kernels.
#include "common.cuh"
#include "kernels.h"

namespace sr {
namespace {

constexpr int BN = 64, BK = 64;

// Shared epilogue of every GEMM variant, applied to one output element.
template <typename T, Epi E>
__device__ __forceinline__ void epilogue_store(const EpiArgs& ea, int m, int n, int N,
                                               float acc) {
  const T* bias = static_cast<const T*>(ea.bias);
  float v = acc + Elem<T>::to_f(bias[n]);
  if constexpr (E == Epi::Bias) {
    static_cast<T*>(ea.out)[size_t(m) * N + n] = Elem<T>::from_f(v);
  } else if constexpr (E == Epi::BiasGelu) {
    static_cast<T*>(ea.out)[size_t(m) * N + n] = Elem<T>::from_f(gelu_erf(v));
  } else if constexpr (E == Epi::BiasResidual) {
    const float r = ea.res[size_t(m) * N + n];
    static_cast<float*>(ea.out)[size_t(m) * N + n] = r + v;
  } else {
    // last sparse block: hn = h + f(h); x'[xrow] = x0 + (hn - h0), h0 == x0
    const float hn = ea.res[size_t(m) * N + n] + v;
    const int b = m / ea.Kr;
    const size_t xrow = size_t(b) * ea.Lx + ea.idx[m];
    float* o = static_cast<float*>(ea.out) + xrow * N + n;
    const float x0 = *o;
    const float delta = hn - x0;
    *o = x0 + delta;
  }
}

// four consecutive elements (16-byte aligned for fp32, 8-byte for bf16) as fp32
__device__ __forceinline__ float4 load4(const float* p) { return __ldg(reinterpret_cast<const float4*>(p)); }
__device__ __forceinline__ float4 load4(const bf16* p) {
  const uint2 u = __ldg(reinterpret_cast<const uint2*>(p));
  return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xffff0000u),
                     __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xffff0000u));
}

// BM x 64 output tile per CTA of 256 threads (BM = 64 or 32: 4 or 2 rows x 4
// columns per thread); the 32-row tile doubles the CTAs of small GEMMs.  The
// next 64-column k-slice of A and W is loaded into registers (4 consecutive k
// per load, 4 loads per matrix and thread) while the current one is multiplied
// from shared memory.
// kPart: split-K; CTA z of the grid's third dimension multiplies the K / gridDim.z
// columns from z * K / gridDim.z on and stores its raw sums in part[z][M][N]
// (the epilogue runs in splitk_epilogue_kernel).
template <typename T, Epi E, int BM, bool kPart = false>
__global__ void __launch_bounds__(256)
gemm_simt_kernel(const T* __restrict__ A, const T* __restrict__ W, int M, int N, int K,
                 EpiArgs ea, float* __restrict__ part = nullptr) {
  constexpr int RI = BM / 16;
  const int Kc = kPart ? K / int(gridDim.z) : K;          // columns of K this CTA multiplies
  const int kz = kPart ? int(blockIdx.z) * Kc : 0;
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int tid = threadIdx.x;
  const int tx = tid & 15, ty = tid >> 4;
  const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
  float acc[RI][4] = {};
  // loader: row lr, k lk + 16u .. lk + 16u + 3 for u = 0..3
  constexpr int kLq = BK / 16;
  const int lr = tid >> 2, lk = (tid & 3) * 4;
  const int am = m0 + lr, bn = n0 + lr;
  const bool a_ok = lr < BM && am < M, b_ok = bn < N;
  const T* ap = A + size_t(a_ok ? am : 0) * K + kz + lk;
  const T* bp = W + size_t(b_ok ? bn : 0) * K + kz + lk;
  const float4 zero = make_float4(0.f, 0.f, 0.f, 0.f);
  float4 ra[kLq], rb[kLq];
#pragma unroll
  for (int u = 0; u < kLq; ++u) {
    ra[u] = a_ok ? load4(ap + 16 * u) : zero;
    rb[u] = b_ok ? load4(bp + 16 * u) : zero;
  }
  for (int k0 = 0; k0 < Kc; k0 += BK) {
#pragma unroll
    for (int u = 0; u < kLq; ++u) {
      const int kk = lk + 16 * u;
      if (lr < BM) {
        As[kk][lr] = ra[u].x; As[kk + 1][lr] = ra[u].y; As[kk + 2][lr] = ra[u].z; As[kk + 3][lr] = ra[u].w;
      }
      Bs[kk][lr] = rb[u].x; Bs[kk + 1][lr] = rb[u].y; Bs[kk + 2][lr] = rb[u].z; Bs[kk + 3][lr] = rb[u].w;
    }
    __syncthreads();
    if (k0 + BK < Kc) {
#pragma unroll
      for (int u = 0; u < kLq; ++u) {
        ra[u] = a_ok ? load4(ap + k0 + BK + 16 * u) : zero;
        rb[u] = b_ok ? load4(bp + k0 + BK + 16 * u) : zero;
      }
    }
#pragma unroll
    for (int k = 0; k < BK; ++k) {
      float a[RI], b[4];
#pragma unroll
      for (int i = 0; i < RI; ++i) a[i] = As[k][ty + 16 * i];
#pragma unroll
      for (int i = 0; i < 4; ++i) b[i] = Bs[k][tx + 16 * i];
#pragma unroll
      for (int i = 0; i < RI; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < RI; ++i) {
    const int m = m0 + ty + 16 * i;
    if (m >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx + 16 * j;
      if (n >= N) continue;
      if constexpr (kPart)
        part[(size_t(blockIdx.z) * M + m) * N + n] = acc[i][j];
      else
        epilogue_store<T, E>(ea, m, n, N, acc[i][j]);
    }
  }
}

// The split-K sums part[0] + part[1] + ... (in slice order) and the fused
// epilogue, one output element per thread.
template <typename T, Epi E>
__global__ void __launch_bounds__(256)
splitk_epilogue_kernel(const float* __restrict__ part, int S, int M, int N, EpiArgs ea) {
  const size_t MN = size_t(M) * N;
  for (size_t i = size_t(blockIdx.x) * blockDim.x + threadIdx.x; i < MN;
       i += size_t(gridDim.x) * blockDim.x) {
    float acc = part[i];
    for (int z = 1; z < S; ++z) acc += part[size_t(z) * MN + i];
    epilogue_store<T, E>(ea, int(i / N), int(i % N), N, acc);
  }
}

// Attention core: 16 query rows per CTA of 128 threads, each row's keys split
// over 8 adjacent lanes (lane p of a row takes keys p, p + 8, ... of every
// tile), keys and values staged in shared memory in tiles of 32, an online
// softmax (running max and sum) per lane in fp32, and the 8 partial states of
// a row merged by shuffles at the end:
//   m = max_p m_p,  l = sum_p l_p 2^(m_p - m),  o = sum_p o_p 2^(m_p - m).
constexpr int kAttRows = 16, kAttParts = 8, kAttThreads = kAttRows * kAttParts;
constexpr int kAttKeys = 32, kDh = 64;

template <typename T>
__global__ void __launch_bounds__(kAttThreads)
attention_simt_kernel(const T* __restrict__ qkv, T* __restrict__ out, int T_, int heads) {
  // rows padded to 68 floats: the 8 keys a warp reads at once (one per lane
  // part) start on 8 different 16-byte bank groups
  __shared__ __align__(16) float Ks[kAttKeys][kDh + 4];
  __shared__ __align__(16) float Vs[kAttKeys][kDh + 4];
  const int D = heads * kDh;
  const int ld = 3 * D;
  const int qtiles = (T_ + kAttRows - 1) / kAttRows;
  const int bh = blockIdx.x / qtiles;
  const int qt = blockIdx.x % qtiles;
  const int b = bh / heads, h = bh % heads;
  const int part = threadIdx.x % kAttParts;
  const int row = qt * kAttRows + threadIdx.x / kAttParts;
  const bool valid = row < T_;
  const T* base = qkv + size_t(b) * T_ * ld;
  // scores in the log2 domain: s * (1/sqrt(64)) * log2(e)
  const float qscale = 0.125f * 1.4426950408889634f;
  float q[kDh], o[kDh];
  {
    const T* qr = base + size_t(valid ? row : 0) * ld + h * kDh;
#pragma unroll
    for (int d = 0; d < kDh; ++d) { q[d] = Elem<T>::to_f(qr[d]) * qscale; o[d] = 0.f; }
  }
  float mrun = -INFINITY, lrun = 0.f;
  constexpr int kMine = kAttKeys / kAttParts;            // keys of a tile per lane
  for (int j0 = 0; j0 < T_; j0 += kAttKeys) {
    __syncthreads();
    // the tile's keys and values, 4 consecutive elements per load; all of a
    // thread's loads are issued before the first store
    constexpr int kQuads = kAttKeys * kDh / 4 / kAttThreads;
    float4 kq[kQuads], vq[kQuads];
#pragma unroll
    for (int u = 0; u < kQuads; ++u) {
      const int e = 4 * (threadIdx.x + u * kAttThreads);
      const int j = e / kDh, d = e % kDh;
      const int key = j0 + j;
      kq[u] = vq[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      if (key < T_) {
        const T* kr = base + size_t(key) * ld + D + h * kDh + d;
        kq[u] = load4(kr);
        vq[u] = load4(kr + D);
      }
    }
#pragma unroll
    for (int u = 0; u < kQuads; ++u) {
      const int e = 4 * (threadIdx.x + u * kAttThreads);
      *reinterpret_cast<float4*>(&Ks[e / kDh][e % kDh]) = kq[u];
      *reinterpret_cast<float4*>(&Vs[e / kDh][e % kDh]) = vq[u];
    }
    __syncthreads();
    float s[kMine];
    float tmax = -INFINITY;
#pragma unroll
    for (int i = 0; i < kMine; ++i) {
      const int j = part + kAttParts * i;
      float acc = 0.f;
#pragma unroll
      for (int d = 0; d < kDh; d += 4) {
        const float4 k4 = *reinterpret_cast<const float4*>(&Ks[j][d]);
        acc = fmaf(q[d], k4.x, acc); acc = fmaf(q[d + 1], k4.y, acc);
        acc = fmaf(q[d + 2], k4.z, acc); acc = fmaf(q[d + 3], k4.w, acc);
      }
      s[i] = (j0 + j < T_) ? acc : -INFINITY;
      tmax = fmaxf(tmax, s[i]);
    }
    // a lane whose keys so far all lie past the end keeps its empty state
    if (tmax == -INFINITY) continue;
    const float mnew = fmaxf(mrun, tmax);
    const float corr = exp2f(mrun - mnew);
    lrun *= corr;
#pragma unroll
    for (int d = 0; d < kDh; ++d) o[d] *= corr;
#pragma unroll
    for (int i = 0; i < kMine; ++i) {
      const int j = part + kAttParts * i;
      const float p = exp2f(s[i] - mnew);
      lrun += p;
#pragma unroll
      for (int d = 0; d < kDh; d += 4) {
        const float4 v4 = *reinterpret_cast<const float4*>(&Vs[j][d]);
        o[d] = fmaf(p, v4.x, o[d]); o[d + 1] = fmaf(p, v4.y, o[d + 1]);
        o[d + 2] = fmaf(p, v4.z, o[d + 2]); o[d + 3] = fmaf(p, v4.w, o[d + 3]);
      }
    }
    mrun = mnew;
  }
  // merge the row's 8 partial states (lanes 8r .. 8r+7 of the warp); every row
  // has at least one key, so the merged max is finite
  float m = mrun;
#pragma unroll
  for (int off = 1; off < kAttParts; off <<= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
  const float w = mrun == -INFINITY ? 0.f : exp2f(mrun - m);
  float l = lrun * w;
#pragma unroll
  for (int off = 1; off < kAttParts; off <<= 1) l += __shfl_xor_sync(0xffffffffu, l, off);
#pragma unroll
  for (int d = 0; d < kDh; ++d) {
    float v = o[d] * w;
#pragma unroll
    for (int off = 1; off < kAttParts; off <<= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    o[d] = v;
  }
  if (valid) {
    // lane p of the row writes dimensions 8p .. 8p + 7
    const float inv = 1.f / l;
    T* orow = out + (size_t(b) * T_ + row) * D + h * kDh;
#pragma unroll
    for (int d = 0; d < kDh; ++d)
      if (d / (kDh / kAttParts) == part) orow[d] = Elem<T>::from_f(o[d] * inv);
  }
}

template <typename T, int BM>
cudaError_t gemm_simt_bm(Epi epi, const void* A, const void* Bw, int M, int N, int K,
                         const EpiArgs& ea, cudaStream_t s) {
  dim3 grid((N + BN - 1) / BN, (M + BM - 1) / BM);
  const T* a = static_cast<const T*>(A);
  const T* w = static_cast<const T*>(Bw);
  switch (epi) {
    case Epi::Bias: gemm_simt_kernel<T, Epi::Bias, BM><<<grid, 256, 0, s>>>(a, w, M, N, K, ea); break;
    case Epi::BiasGelu:
      gemm_simt_kernel<T, Epi::BiasGelu, BM><<<grid, 256, 0, s>>>(a, w, M, N, K, ea); break;
    case Epi::BiasResidual:
      gemm_simt_kernel<T, Epi::BiasResidual, BM><<<grid, 256, 0, s>>>(a, w, M, N, K, ea); break;
    case Epi::BiasResidualScatter:
      gemm_simt_kernel<T, Epi::BiasResidualScatter, BM><<<grid, 256, 0, s>>>(a, w, M, N, K, ea);
      break;
  }
  return cudaGetLastError();
}

template <typename T, Epi E>
cudaError_t gemm_simt_splitk(const T* a, const T* w, int M, int N, int K, int S,
                             const EpiArgs& ea, float* part, cudaStream_t s) {
  dim3 grid((N + BN - 1) / BN, (M + 31) / 32, S);
  gemm_simt_kernel<T, E, 32, true><<<grid, 256, 0, s>>>(a, w, M, N, K, ea, part);
  const size_t MN = size_t(M) * N;
  const int blocks = int((MN + 255) / 256 < 152 * 8 ? (MN + 255) / 256 : 152 * 8);
  splitk_epilogue_kernel<T, E><<<blocks, 256, 0, s>>>(part, S, M, N, ea);
  return cudaGetLastError();
}

template <typename T>
cudaError_t gemm_simt_t(Epi epi, const void* A, const void* Bw, int M, int N, int K,
                        const EpiArgs& ea, cudaStream_t s, float* part, size_t part_floats) {
  // 64-row tiles when they already give two CTAs per SM, else 32-row tiles;
  // when even those leave SMs idle, K is split into S slices (a power of two,
  // at most 8, each at least 128 columns) that run side by side
  const long ctas64 = long((N + BN - 1) / BN) * ((M + 63) / 64);
  if (ctas64 >= 2 * 152) return gemm_simt_bm<T, 64>(epi, A, Bw, M, N, K, ea, s);
  const long ctas32 = long((N + BN - 1) / BN) * ((M + 31) / 32);
  int S = 1;
  while (ctas32 * S < 2 * 152 && S < 8 && K % (2 * S * BK) == 0 && K / (2 * S) >= 128) S *= 2;
  if (S > 1 && part && size_t(S) * M * N <= part_floats) {
    const T* a = static_cast<const T*>(A);
    const T* w = static_cast<const T*>(Bw);
    switch (epi) {
      case Epi::Bias: return gemm_simt_splitk<T, Epi::Bias>(a, w, M, N, K, S, ea, part, s);
      case Epi::BiasGelu: return gemm_simt_splitk<T, Epi::BiasGelu>(a, w, M, N, K, S, ea, part, s);
      case Epi::BiasResidual:
        return gemm_simt_splitk<T, Epi::BiasResidual>(a, w, M, N, K, S, ea, part, s);
      case Epi::BiasResidualScatter:
        return gemm_simt_splitk<T, Epi::BiasResidualScatter>(a, w, M, N, K, S, ea, part, s);
    }
  }
  return gemm_simt_bm<T, 32>(epi, A, Bw, M, N, K, ea, s);
}

}  // namespace

cudaError_t launch_gemm_simt(DType dt, Epi epi, const void* A, const void* Bw, int M, int N,
                             int K, const EpiArgs& ea, cudaStream_t s, float* splitk,
                             size_t splitk_floats) {
  if (ea.sqnorm) return cudaErrorInvalidValue;     // row norms are fused on the tcgen05 path only
  if (dt == DType::F32) return gemm_simt_t<float>(epi, A, Bw, M, N, K, ea, s, splitk, splitk_floats);
  return gemm_simt_t<bf16>(epi, A, Bw, M, N, K, ea, s, splitk, splitk_floats);
}

cudaError_t launch_attention_simt(DType dt, const void* qkv, void* out, int B, int T, int heads,
                                  cudaStream_t s) {
  const int grid = B * heads * ((T + kAttRows - 1) / kAttRows);
  if (dt == DType::F32)
    attention_simt_kernel<float><<<grid, kAttThreads, 0, s>>>(static_cast<const float*>(qkv),
                                                              static_cast<float*>(out), T, heads);
  else
    attention_simt_kernel<bf16><<<grid, kAttThreads, 0, s>>>(static_cast<const bf16*>(qkv),
                                                             static_cast<bf16*>(out), T, heads);
  return cudaGetLastError();
}

}  // namespace sr
