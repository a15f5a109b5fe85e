// Row-wise HBM-bound kernels on the fp32 residual stream: LayerNorm (the LN of
// the pre-LN block, Sec. 3.3 Eq. 11), which for the first sparse block also
// performs the routed-token gather (Eq. 8) through the index set; the
// conversions between the caller's storage dtype and the stream; and the
// implicit ensemble's copies of the dense-early result and mean of its members.
// In LayerNorm one warp owns one row; rows move as 16-byte vectors, all loads
// of a row are issued before any use.
#include "common.cuh"
#include "kernels.h"

namespace sr {
namespace {

// y = (x - mean) / sqrt(var + eps) * g + b from the fp32 stream x into the
// storage dtype T, statistics in fp32, two passes over the row held in
// registers (biased variance).  Rows are read as 4-float vectors, g, b and y
// move as 16-byte vectors of T.
// With idx set, this is LN1 of the first sparse block fused with the gather
// of Eq. 8: output row r (sample r / K) normalises stream row (r / K) * L +
// idx[r], and that fp32 row is also copied to hcopy[r] (h0, the start of the
// routed stream).
template <typename T, int NV>
__global__ void __launch_bounds__(256)
layernorm_kernel(const float* __restrict__ x, const T* __restrict__ g, const T* __restrict__ bta,
                 T* __restrict__ y, int rows, int D, float eps, const int32_t* __restrict__ idx,
                 int L, int K, float* __restrict__ hcopy) {
  pdl_wait();      // the previous kernel's writes are visible from here
  pdl_trigger();
  constexpr int V = Elem<T>::kVec;
  const int lane = threadIdx.x & 31;
  const int row = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (row >= rows) return;
  const int nv = D / V;
  const size_t src = idx ? size_t(row / K) * L + size_t(__ldg(idx + row)) : size_t(row);
  const float4* xr = reinterpret_cast<const float4*>(x + src * D);
  float f[NV][V];
  float sum = 0.f;
#pragma unroll
  for (int j = 0; j < NV; ++j) {
    if (lane + 32 * j < nv) {
#pragma unroll
      for (int q = 0; q < V / 4; ++q) {
        const float4 v4 = __ldg(xr + (lane + 32 * j) * (V / 4) + q);
        f[j][4 * q] = v4.x; f[j][4 * q + 1] = v4.y; f[j][4 * q + 2] = v4.z; f[j][4 * q + 3] = v4.w;
      }
#pragma unroll
      for (int e = 0; e < V; ++e) sum += f[j][e];
    }
  }
  const float inv_d = 1.0f / float(D);
  const float mean = warp_sum(sum) * inv_d;
  float sq = 0.f;
#pragma unroll
  for (int j = 0; j < NV; ++j) {
    if (lane + 32 * j < nv) {
#pragma unroll
      for (int e = 0; e < V; ++e) { const float c = f[j][e] - mean; sq = fmaf(c, c, sq); }
    }
  }
  const float rstd = rsqrtf(warp_sum(sq) * inv_d + eps);
  if (hcopy) {
    float4* hr = reinterpret_cast<float4*>(hcopy + size_t(row) * D);
#pragma unroll
    for (int j = 0; j < NV; ++j)
      if (lane + 32 * j < nv)
#pragma unroll
        for (int q = 0; q < V / 4; ++q)
          hr[(lane + 32 * j) * (V / 4) + q] =
              make_float4(f[j][4 * q], f[j][4 * q + 1], f[j][4 * q + 2], f[j][4 * q + 3]);
  }
  const uint4* gr = reinterpret_cast<const uint4*>(g);
  const uint4* br = reinterpret_cast<const uint4*>(bta);
  uint4* yr = reinterpret_cast<uint4*>(y + size_t(row) * D);
#pragma unroll
  for (int j = 0; j < NV; ++j) {
    const int v = lane + 32 * j;
    if (v < nv) {
      float gf[V], bf[V], o[V];
      unpack16(__ldg(gr + v), gf);
      unpack16(__ldg(br + v), bf);
#pragma unroll
      for (int e = 0; e < V; ++e) o[e] = (f[j][e] - mean) * rstd * gf[e] + bf[e];
      yr[v] = pack16(o);
    }
  }
}

// Storage dtype <-> fp32 stream, n elements (n % 8 == 0), 16-byte vectors.
template <typename T>
__global__ void __launch_bounds__(256)
widen_kernel(const T* __restrict__ x, float* __restrict__ y, size_t nvec, float* zero, int nzero) {
  pdl_wait();      // the previous kernel's writes are visible from here
  pdl_trigger();
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < nzero; i += gridDim.x * blockDim.x)
    zero[i] = 0.f;
  constexpr int V = Elem<T>::kVec;
  for (size_t i = size_t(blockIdx.x) * blockDim.x + threadIdx.x; i < nvec;
       i += size_t(gridDim.x) * blockDim.x) {
    float f[V];
    unpack16(__ldg(reinterpret_cast<const uint4*>(x) + i), f);
    float4* o = reinterpret_cast<float4*>(y) + i * (V / 4);
#pragma unroll
    for (int q = 0; q < V / 4; ++q) o[q] = make_float4(f[4 * q], f[4 * q + 1], f[4 * q + 2], f[4 * q + 3]);
  }
}

// y[m] = x for m = 0 .. M-1 (the implicit ensemble's members start from the
// same dense-early result), 4-float vectors
__global__ void __launch_bounds__(256)
replicate_kernel(const float* __restrict__ x, float* __restrict__ y, size_t nvec, int M) {
  pdl_wait();      // the previous kernel's writes are visible from here
  pdl_trigger();
  const float4* xv = reinterpret_cast<const float4*>(x);
  float4* yv = reinterpret_cast<float4*>(y);
  for (size_t i = size_t(blockIdx.x) * blockDim.x + threadIdx.x; i < nvec;
       i += size_t(gridDim.x) * blockDim.x) {
    const float4 v = __ldg(xv + i);
    for (int m = 0; m < M; ++m) yv[size_t(m) * nvec + i] = v;
  }
}

// y = scale * (x[0] + x[1] + ... + x[M-1]) rounded once to the storage dtype T,
// the sum in fp32 in member order (x: M consecutive fp32 streams of nvec vectors)
template <typename T>
__global__ void __launch_bounds__(256)
mean_narrow_kernel(const float* __restrict__ x, int M, size_t nvec, float scale, T* __restrict__ y) {
  pdl_wait();      // the previous kernel's writes are visible from here
  pdl_trigger();
  constexpr int V = Elem<T>::kVec;
  const size_t n4 = nvec * (V / 4);            // float4 vectors per member
  for (size_t i = size_t(blockIdx.x) * blockDim.x + threadIdx.x; i < nvec;
       i += size_t(gridDim.x) * blockDim.x) {
    float f[V];
    const float4* in = reinterpret_cast<const float4*>(x) + i * (V / 4);
#pragma unroll
    for (int q = 0; q < V / 4; ++q) {
      const float4 v4 = __ldg(in + q);
      f[4 * q] = v4.x; f[4 * q + 1] = v4.y; f[4 * q + 2] = v4.z; f[4 * q + 3] = v4.w;
    }
    for (int m = 1; m < M; ++m) {
#pragma unroll
      for (int q = 0; q < V / 4; ++q) {
        const float4 v4 = __ldg(in + size_t(m) * n4 + q);
        f[4 * q] += v4.x; f[4 * q + 1] += v4.y; f[4 * q + 2] += v4.z; f[4 * q + 3] += v4.w;
      }
    }
#pragma unroll
    for (int e = 0; e < V; ++e) f[e] *= scale;
    reinterpret_cast<uint4*>(y)[i] = pack16(f);
  }
}

template <typename T>
__global__ void __launch_bounds__(256)
narrow_kernel(const float* __restrict__ x, T* __restrict__ y, size_t nvec, float scale) {
  pdl_wait();      // the previous kernel's writes are visible from here
  pdl_trigger();
  constexpr int V = Elem<T>::kVec;
  for (size_t i = size_t(blockIdx.x) * blockDim.x + threadIdx.x; i < nvec;
       i += size_t(gridDim.x) * blockDim.x) {
    float f[V];
    const float4* in = reinterpret_cast<const float4*>(x) + i * (V / 4);
#pragma unroll
    for (int q = 0; q < V / 4; ++q) {
      const float4 v4 = __ldg(in + q);
      f[4 * q] = v4.x * scale; f[4 * q + 1] = v4.y * scale;
      f[4 * q + 2] = v4.z * scale; f[4 * q + 3] = v4.w * scale;
    }
    reinterpret_cast<uint4*>(y)[i] = pack16(f);
  }
}

int grid_for(size_t nvec) {
  size_t b = (nvec + 255) / 256;
  return int(b < 152 * 32 ? b : 152 * 32);
}

template <typename T, int NV>
cudaError_t layernorm_t(const float* x, const void* g, const void* b, void* y, int rows, int D,
                        float eps, cudaStream_t s, const int32_t* idx, int L, int K, float* hcopy) {
  return launch_k(layernorm_kernel<T, NV>, dim3((rows + 7) / 8), dim3(256), 0, s, 1, x,
                  static_cast<const T*>(g), static_cast<const T*>(b), static_cast<T*>(y), rows, D,
                  eps, idx, L, K, hcopy);
}

// vectors per lane needed for a row of D elements
template <typename T> int lanes_nv(int D) { return (D / Elem<T>::kVec + 31) / 32; }

}  // namespace

cudaError_t launch_widen(DType dt, const void* x, float* y, size_t n, cudaStream_t s,
                         float* zero, int nzero) {
  if (!zero) nzero = 0;
  if (dt == DType::BF16) {
    const size_t nvec = n / 8;
    return launch_k(widen_kernel<bf16>, dim3(grid_for(nvec)), dim3(256), 0, s, 1,
                    static_cast<const bf16*>(x), y, nvec, zero, nzero);
  }
  const size_t nvec = n / 4;
  return launch_k(widen_kernel<float>, dim3(grid_for(nvec)), dim3(256), 0, s, 1,
                  static_cast<const float*>(x), y, nvec, zero, nzero);
}

cudaError_t launch_narrow(DType dt, const float* x, void* y, size_t n, cudaStream_t s, float scale) {
  if (dt == DType::BF16) {
    const size_t nvec = n / 8;
    return launch_k(narrow_kernel<bf16>, dim3(grid_for(nvec)), dim3(256), 0, s, 1, x,
                    static_cast<bf16*>(y), nvec, scale);
  }
  const size_t nvec = n / 4;
  return launch_k(narrow_kernel<float>, dim3(grid_for(nvec)), dim3(256), 0, s, 1, x,
                  static_cast<float*>(y), nvec, scale);
}

cudaError_t launch_replicate(const float* x, float* y, size_t n, int M, cudaStream_t s) {
  const size_t nvec = n / 4;
  return launch_k(replicate_kernel, dim3(grid_for(nvec)), dim3(256), 0, s, 1, x, y, nvec, M);
}

cudaError_t launch_mean_narrow(DType dt, const float* x, int M, size_t n, float scale, void* y,
                               cudaStream_t s) {
  if (dt == DType::BF16) {
    const size_t nvec = n / 8;
    return launch_k(mean_narrow_kernel<bf16>, dim3(grid_for(nvec)), dim3(256), 0, s, 1, x, M, nvec,
                    scale, static_cast<bf16*>(y));
  }
  const size_t nvec = n / 4;
  return launch_k(mean_narrow_kernel<float>, dim3(grid_for(nvec)), dim3(256), 0, s, 1, x, M, nvec,
                  scale, static_cast<float*>(y));
}

cudaError_t launch_layernorm(DType dt, const float* x, const void* g, const void* b, void* y,
                             int rows, int D, float eps, cudaStream_t s, const int32_t* idx,
                             int L, int K, float* hcopy) {
  if (dt == DType::BF16) {
    const int nv = lanes_nv<bf16>(D);
    if (nv <= 1) return layernorm_t<bf16, 1>(x, g, b, y, rows, D, eps, s, idx, L, K, hcopy);
    if (nv <= 2) return layernorm_t<bf16, 2>(x, g, b, y, rows, D, eps, s, idx, L, K, hcopy);
    if (nv <= 4) return layernorm_t<bf16, 4>(x, g, b, y, rows, D, eps, s, idx, L, K, hcopy);
    if (nv <= 8) return layernorm_t<bf16, 8>(x, g, b, y, rows, D, eps, s, idx, L, K, hcopy);
  } else {
    const int nv = lanes_nv<float>(D);
    if (nv <= 1) return layernorm_t<float, 1>(x, g, b, y, rows, D, eps, s, idx, L, K, hcopy);
    if (nv <= 2) return layernorm_t<float, 2>(x, g, b, y, rows, D, eps, s, idx, L, K, hcopy);
    if (nv <= 4) return layernorm_t<float, 4>(x, g, b, y, rows, D, eps, s, idx, L, K, hcopy);
    if (nv <= 8) return layernorm_t<float, 8>(x, g, b, y, rows, D, eps, s, idx, L, K, hcopy);
  }
  return cudaErrorInvalidValue;
}

}  // namespace sr
