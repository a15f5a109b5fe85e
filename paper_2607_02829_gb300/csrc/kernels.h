// Internal launchers of the Sparse-Reslim CUDA library.  Every launcher only
// enqueues work on `stream` and returns the launch's cudaError_t.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace sr {

enum class DType : int { F32 = 0, BF16 = 1 };

// ---- programmatic dependent launch -----------------------------------------
// While a PdlScope is alive on the calling thread, the launchers below mark
// each kernel as allowed to start while the previous kernel of the stream is
// still finishing.  Such a kernel runs its setup (barriers, tensor memory,
// tensor-map prefetch) early, and every thread waits (griddepcontrol.wait)
// for the previous grids to complete before it touches global memory.
bool pdl_enabled();
struct PdlScope {
  explicit PdlScope(bool on);
  ~PdlScope();
  PdlScope(const PdlScope&) = delete;
  PdlScope& operator=(const PdlScope&) = delete;
  bool prev;
};
template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                            cudaStream_t s, unsigned cluster, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cudaLaunchAttribute at[2];
  unsigned n = 0;
  if (pdl_enabled()) {
    at[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  if (cluster > 1) {
    at[n].id = cudaLaunchAttributeClusterDimension;
    at[n].val.clusterDim.x = cluster;
    at[n].val.clusterDim.y = 1;
    at[n].val.clusterDim.z = 1;
    ++n;
  }
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = at;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

// ---- per-device caches of launch attributes -------------------------------
// Kernel shared-memory limits and occupancy belong to a device's context, so
// the launchers cache them per device ordinal (the current device).  Returns
// -1 when the current device cannot be read or its ordinal is 64 or more.
constexpr int kMaxDevices = 64;
inline int device_slot() {
  int d = 0;
  if (cudaGetDevice(&d) != cudaSuccess || d < 0 || d >= kMaxDevices) return -1;
  return d;
}

// ---- token selection (Sec. 3.2; App. B.2) --------------------------------
// Random: K smallest SplitMix64 keys per sample (ties by index), sorted indices.
cudaError_t launch_select_random(int B, int L, int K, uint64_t seed, int shared,
                                 int32_t* idx, cudaStream_t s);
// Squared L2 norm of every token of the fp32 stream x [B*L, D] into score [B*L];
// each value is first rounded to the storage dtype dt (the activation the model
// stores), its square accumulated in fp32.
cudaError_t launch_token_sq_norms(DType dt, const float* x, int rows, int D, float* score,
                                  cudaStream_t s);
// Laplacian score of every token of the fp32 stream x [B*L, D] into score [B*L]:
// tokens row-major on a patch grid grid_w wide, 5-point stencil with periodic
// longitude and the first and last rows reflected; each value rounded to the
// storage dtype dt, the squared norm of the stencil accumulated in fp32.
cudaError_t launch_token_laplacian(DType dt, const float* x, int B, int L, int grid_w, int D,
                                   float* score, cudaStream_t s);
// K largest scores per sample (ties to the lower index), sorted indices.  A
// token's score is the sum of `parts` consecutive partial sums (score
// [B*L][parts]), added in order.
cudaError_t launch_select_topk(int B, int L, int K, const float* score, int32_t* idx,
                               cudaStream_t s, int parts = 1);
// Largest L the one-CTA-per-sample selection kernels accept (keys in shared memory).
int select_max_L();

// ---- storage dtype <-> fp32 residual stream, n elements (n % 8 == 0) ------
// also zeroes zero[0, nzero) when given
cudaError_t launch_widen(DType dt, const void* x, float* y, size_t n, cudaStream_t s,
                         float* zero = nullptr, int nzero = 0);
// narrow rounds scale * x once to the storage dtype
cudaError_t launch_narrow(DType dt, const float* x, void* y, size_t n, cudaStream_t s,
                          float scale = 1.0f);
// y[m * n + i] = x[i] for m < M, fp32, n % 4 == 0
cudaError_t launch_replicate(const float* x, float* y, size_t n, int M, cudaStream_t s);
// y = scale * sum_m x[m * n + i] rounded once to the storage dtype, the sum in
// fp32 in member order, n % 8 == 0
cudaError_t launch_mean_narrow(DType dt, const float* x, int M, size_t n, float scale, void* y,
                               cudaStream_t s);

// ---- LayerNorm over D from the fp32 stream into the storage dtype ---------
//      y = (x - mean) / sqrt(var + eps) * g + b
//      With idx set (LN1 of the first sparse block fused with the gather of
//      Eq. 8): row r reads stream row (r / K) * L + idx[r] and also copies that
//      fp32 row to hcopy[r].
cudaError_t launch_layernorm(DType dt, const float* x, const void* g, const void* b, void* y,
                             int rows, int D, float eps, cudaStream_t s,
                             const int32_t* idx = nullptr, int L = 0, int K = 0,
                             float* hcopy = nullptr);

// ---- GEMM C = A B^T with fused epilogues ---------------------------------
// A [M, K] row-major, B [N, K] row-major (nn.Linear weight), both in the storage
// dtype, fp32 accumulate.  Bias is in the storage dtype.
enum class Epi : int {
  Bias = 0,          // out[m, n] = acc + bias[n]                   (out: storage dtype)
  BiasGelu = 1,      // out[m, n] = GELU(acc + bias[n])             (out: storage dtype)
  BiasResidual = 2,  // out[m, n] = res[m, n] + acc + bias[n]       (fp32 stream, out may == res)
  BiasResidualScatter = 3,  // hn = res[m, n] + acc + bias[n] (fp32 routed stream); row
                            // m = b*Kr + k maps to xrow = b*Lx + idx[m]; the fp32 stream
                            // out[xrow, n] = x0 + (hn - x0) with x0 = out[xrow, n]
};
struct EpiArgs {
  const void* bias;     // [N]
  const float* res;     // [M, N] fp32 stream (BiasResidual*)
  void* out;            // [M, N], or the fp32 stream [B*Lx, N] for the scatter epilogue
  const int32_t* idx;   // [M] for the scatter epilogue
  int Kr;               // routed rows per sample (scatter)
  int Lx;               // tokens per sample of the scatter target
  unsigned int* fault;  // fault word (bit 0: a bounded barrier wait timed out)
  float* sqnorm;        // [M][2N/BN] optional (BiasResidual on pair tiles): per row, one sum
                        // of squares of the updated values (each rounded to bf16 first)
                        // for each half tile of BN/2 columns, in column order
};
// CUDA-core GEMM (fp32 storage) and tcgen05 GEMM (bf16 storage; K % 64 == 0,
// N % 64 == 0).
// splitk: optional fp32 scratch of splitk_floats for the partial sums of a
// split-K launch (used when the output tiles alone would leave SMs idle).
cudaError_t launch_gemm_simt(DType dt, Epi epi, const void* A, const void* Bw, int M, int N,
                             int K, const EpiArgs& ea, cudaStream_t s, float* splitk = nullptr,
                             size_t splitk_floats = 0);
cudaError_t launch_gemm_tc(Epi epi, const void* A, const void* Bw, int M, int N, int K,
                           const EpiArgs& ea, cudaStream_t s);
// partial sums per row that launch_gemm_tc writes to EpiArgs::sqnorm for a
// BiasResidual GEMM N columns wide; 0 when it does not take sqnorm
int gemm_tc_sqnorm_parts(int N);


// ---- attention core: per (sample, head) softmax(q k^T / sqrt(64)) v ------
// qkv [B*T, 3D] (q | k | v, head h at columns 64h..64h+63 of each); out [B*T, D].
// CUDA-core version (fp32 storage) and tcgen05 version (bf16 storage).
cudaError_t launch_attention_simt(DType dt, const void* qkv, void* out, int B, int T, int heads,
                                  cudaStream_t s);
cudaError_t launch_attention_tc(const void* qkv, void* out, int B, int T, int heads,
                                unsigned int* fault, cudaStream_t s);
// Queries and keys/values from different token sets: q [B*Tq, D], kv [B*Tkv, 2D]
// (k | v), out [B*Tq, D]; the same kernel with two tensor maps (bf16).
cudaError_t launch_cross_attention_tc(const void* q, const void* kv, void* out, int B, int Tq,
                                      int Tkv, int heads, unsigned int* fault, cudaStream_t s);

}  // namespace sr
