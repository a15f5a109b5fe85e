// CUDA-core (FFMA) kernels for the fp32 configuration: the block GEMMs with
// their fused epilogues and the attention core.  fp32 end to end, because TF32
// tensor cores would not hold the fp32 tolerance.  These kernels serve the
// small fp32 model (D = 256); the bf16 path runs on the tcgen05 kernels.
#include "common.cuh"
#include "kernels.h"

namespace sr {
namespace {

constexpr int BM = 64, BN = 64, BK = 16;

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

template <typename T, Epi E>
__global__ void __launch_bounds__(256)
gemm_simt_kernel(const T* __restrict__ A, const T* __restrict__ W, int M, int N, int K,
                 EpiArgs ea) {
  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int tid = threadIdx.x;
  const int tx = tid & 15, ty = tid >> 4;
  const int m0 = blockIdx.y * BM, n0 = blockIdx.x * BN;
  float acc[4][4] = {};
  const int lr = tid >> 2, lk = (tid & 3) * 4;   // loader: row lr, k lk..lk+3
  for (int k0 = 0; k0 < K; k0 += BK) {
    const int am = m0 + lr, bn = n0 + lr;
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      As[lk + e][lr] = am < M ? Elem<T>::to_f(A[size_t(am) * K + k0 + lk + e]) : 0.f;
      Bs[lk + e][lr] = bn < N ? Elem<T>::to_f(W[size_t(bn) * K + k0 + lk + e]) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < BK; ++k) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) { a[i] = As[k][ty + 16 * i]; b[i] = Bs[k][tx + 16 * i]; }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int m = m0 + ty + 16 * i;
    if (m >= M) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + tx + 16 * j;
      if (n < N) epilogue_store<T, E>(ea, m, n, N, acc[i][j]);
    }
  }
}

// Attention core, one query row per thread, 128 rows per CTA, keys in tiles of
// 32 staged in shared memory, online softmax (running max and sum) in fp32.
constexpr int kAttRows = 128, kAttKeys = 32, kDh = 64;

template <typename T>
__global__ void __launch_bounds__(kAttRows)
attention_simt_kernel(const T* __restrict__ qkv, T* __restrict__ out, int T_, int heads) {
  __shared__ __align__(16) float Ks[kAttKeys][kDh];
  __shared__ __align__(16) float Vs[kAttKeys][kDh];
  const int D = heads * kDh;
  const int ld = 3 * D;
  const int qtiles = (T_ + kAttRows - 1) / kAttRows;
  const int bh = blockIdx.x / qtiles;
  const int qt = blockIdx.x % qtiles;
  const int b = bh / heads, h = bh % heads;
  const int row = qt * kAttRows + threadIdx.x;
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
  for (int j0 = 0; j0 < T_; j0 += kAttKeys) {
    __syncthreads();
    for (int e = threadIdx.x; e < kAttKeys * kDh; e += kAttRows) {
      const int j = e / kDh, d = e % kDh;
      const int key = j0 + j;
      float kv = 0.f, vv = 0.f;
      if (key < T_) {
        const T* kr = base + size_t(key) * ld + D + h * kDh;
        kv = Elem<T>::to_f(kr[d]);
        vv = Elem<T>::to_f(kr[D + d]);
      }
      Ks[j][d] = kv;
      Vs[j][d] = vv;
    }
    __syncthreads();
    float s[kAttKeys];
    float tmax = -INFINITY;
#pragma unroll
    for (int j = 0; j < kAttKeys; ++j) {
      float acc = 0.f;
#pragma unroll
      for (int d = 0; d < kDh; d += 4) {
        const float4 k4 = *reinterpret_cast<const float4*>(&Ks[j][d]);
        acc = fmaf(q[d], k4.x, acc); acc = fmaf(q[d + 1], k4.y, acc);
        acc = fmaf(q[d + 2], k4.z, acc); acc = fmaf(q[d + 3], k4.w, acc);
      }
      s[j] = (j0 + j < T_) ? acc : -INFINITY;
      tmax = fmaxf(tmax, s[j]);
    }
    const float mnew = fmaxf(mrun, tmax);
    const float corr = exp2f(mrun - mnew);
    lrun *= corr;
#pragma unroll
    for (int d = 0; d < kDh; ++d) o[d] *= corr;
#pragma unroll
    for (int j = 0; j < kAttKeys; ++j) {
      const float p = exp2f(s[j] - mnew);
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
  if (valid) {
    const float inv = 1.f / lrun;
    T* orow = out + (size_t(b) * T_ + row) * D + h * kDh;
#pragma unroll
    for (int d = 0; d < kDh; ++d) orow[d] = Elem<T>::from_f(o[d] * inv);
  }
}

template <typename T>
cudaError_t gemm_simt_t(Epi epi, const void* A, const void* Bw, int M, int N, int K,
                        const EpiArgs& ea, cudaStream_t s) {
  dim3 grid((N + BN - 1) / BN, (M + BM - 1) / BM);
  const T* a = static_cast<const T*>(A);
  const T* w = static_cast<const T*>(Bw);
  switch (epi) {
    case Epi::Bias: gemm_simt_kernel<T, Epi::Bias><<<grid, 256, 0, s>>>(a, w, M, N, K, ea); break;
    case Epi::BiasGelu: gemm_simt_kernel<T, Epi::BiasGelu><<<grid, 256, 0, s>>>(a, w, M, N, K, ea); break;
    case Epi::BiasResidual: gemm_simt_kernel<T, Epi::BiasResidual><<<grid, 256, 0, s>>>(a, w, M, N, K, ea); break;
    case Epi::BiasResidualScatter:
      gemm_simt_kernel<T, Epi::BiasResidualScatter><<<grid, 256, 0, s>>>(a, w, M, N, K, ea); break;
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemm_simt(DType dt, Epi epi, const void* A, const void* Bw, int M, int N,
                             int K, const EpiArgs& ea, cudaStream_t s) {
  if (ea.sqnorm) return cudaErrorInvalidValue;     // row norms are fused on the tcgen05 path only
  if (dt == DType::F32) return gemm_simt_t<float>(epi, A, Bw, M, N, K, ea, s);
  return gemm_simt_t<bf16>(epi, A, Bw, M, N, K, ea, s);
}

cudaError_t launch_attention_simt(DType dt, const void* qkv, void* out, int B, int T, int heads,
                                  cudaStream_t s) {
  const int grid = B * heads * ((T + kAttRows - 1) / kAttRows);
  if (dt == DType::F32)
    attention_simt_kernel<float><<<grid, kAttRows, 0, s>>>(static_cast<const float*>(qkv),
                                                           static_cast<float*>(out), T, heads);
  else
    attention_simt_kernel<bf16><<<grid, kAttRows, 0, s>>>(static_cast<const bf16*>(qkv),
                                                          static_cast<bf16*>(out), T, heads);
  return cudaGetLastError();
}

}  // namespace sr
