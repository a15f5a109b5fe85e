// Allocation-free top-K L2-norm token selection (sr_select_topk_l2_static).
//
// Same result as sr_select with SR_SEL_TOPK_L2, for callers that cannot
// allocate device memory: the per-token score buffer lives in a file-scope
// static __device__ array instead of a caller-provided workspace.  The array
// is sized for kStaticScoreTokens tokens (B * L) and stays resident on every
// GPU that loads this library until the process exits.
#include <string>

#include "../../include/sparse_reslim.h"
#include "common.cuh"
#include "kernels.h"

namespace sr {
void set_error_message(const std::string& msg);
}  // namespace sr

namespace {

constexpr size_t kStaticScoreTokens = size_t(1) << 20;          // 1,048,576 tokens, 4 MiB
static __device__ __align__(256) float g_static_scores[kStaticScoreTokens];

// One warp per token: squared L2 norm of the stored row, in the same element
// order and with the same fp32 accumulation as the workspace path (4 elements
// per lane step, a warp-wide sum at the end).
template <typename T>
__global__ void __launch_bounds__(256)
stored_sq_norms_kernel(const T* __restrict__ x, int rows, int D, float* __restrict__ score) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= rows) return;
  const T* row = x + size_t(warp) * D;
  float acc = 0.f;
  for (int v = lane; v < D / 4; v += 32) {
    float f[4];
    if constexpr (sizeof(T) == 2) {
      const uint2 u = __ldg(reinterpret_cast<const uint2*>(row) + v);
      f[0] = __uint_as_float(u.x << 16); f[1] = __uint_as_float(u.x & 0xffff0000u);
      f[2] = __uint_as_float(u.y << 16); f[3] = __uint_as_float(u.y & 0xffff0000u);
    } else {
      const float4 q = __ldg(reinterpret_cast<const float4*>(row) + v);
      f[0] = q.x; f[1] = q.y; f[2] = q.z; f[3] = q.w;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) acc = fmaf(f[j], f[j], acc);
  }
  acc = sr::warp_sum(acc);
  if (lane == 0) score[warp] = acc;
}

sr_status reject(sr_status st, const std::string& msg) {
  sr::set_error_message(msg);
  return st;
}

// The device address of the static score array in the current device's context.
// It is looked up on every call (cudaGetSymbolAddress allocates nothing), so a
// context that was reset or recreated since an earlier call is never handed a
// stale address.
sr_status scores_on_current_device(float** out) {
  float* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(reinterpret_cast<void**>(&p), g_static_scores);
  if (e != cudaSuccess || !p)
    return reject(SR_ERR_CUDA, std::string("cudaGetSymbolAddress(static scores): ") +
                                   cudaGetErrorString(e));
  *out = p;
  return SR_OK;
}

}  // namespace

extern "C" sr_status sr_select_topk_l2_static(const void* x, int32_t B, int32_t L, int32_t D,
                                              int32_t dtype, float keep_ratio, int32_t* idx,
                                              int32_t* K_out, void* stream) {
  if (!x || (reinterpret_cast<uintptr_t>(x) % 16) != 0)
    return reject(SR_ERR_INVALID_ARG, "x must be non-NULL and 16-byte aligned");
  if (!idx || (reinterpret_cast<uintptr_t>(idx) % 4) != 0)
    return reject(SR_ERR_INVALID_ARG, "idx must be non-NULL and 4-byte aligned");
  if (dtype != SR_F32 && dtype != SR_BF16) return reject(SR_ERR_INVALID_ARG, "bad dtype");
  if (B < 1 || L < 1) return reject(SR_ERR_INVALID_ARG, "B and L must be >= 1");
  if (D < 64 || D % 64 != 0 || D > (dtype == SR_BF16 ? 2048 : 1024))
    return reject(SR_ERR_UNSUPPORTED, "D must be a multiple of 64 up to 2048 (bf16) / 1024 (fp32)");
  if (L > sr::select_max_L())
    return reject(SR_ERR_UNSUPPORTED, "L exceeds the selection kernel's shared-memory capacity");
  if (size_t(B) * size_t(L) > kStaticScoreTokens)
    return reject(SR_ERR_UNSUPPORTED,
                  "B * L exceeds the static score buffer of 1048576 tokens; use sr_select");
  if (!(keep_ratio > 0.0f) || !(keep_ratio <= 1.0f))
    return reject(SR_ERR_INVALID_ARG, "keep_ratio must lie in (0, 1]");
  const int32_t K = static_cast<int32_t>(double(keep_ratio) * double(L));
  if (K < 1) return reject(SR_ERR_INVALID_ARG, "K = floor(L * keep_ratio) is 0");
  float* scores = nullptr;
  sr_status st = scores_on_current_device(&scores);
  if (st != SR_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const int rows = B * L;
  // every score the selection reads is written first: nothing needs zeroing
  if (dtype == SR_BF16)
    stored_sq_norms_kernel<sr::bf16><<<(rows + 7) / 8, 256, 0, s>>>(
        static_cast<const sr::bf16*>(x), rows, D, scores);
  else
    stored_sq_norms_kernel<float><<<(rows + 7) / 8, 256, 0, s>>>(static_cast<const float*>(x),
                                                                 rows, D, scores);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return reject(SR_ERR_CUDA, std::string("norms: ") + cudaGetErrorString(e));
  e = sr::launch_select_topk(B, L, K, scores, idx, s);
  if (e != cudaSuccess) return reject(SR_ERR_CUDA, std::string("select_topk: ") + cudaGetErrorString(e));
  if (K_out) *K_out = K;
  return SR_OK;
}
