// C ABI of the Sparse-Reslim encoder forward: validation, workspace carve-up and
// the launch sequence of Alg. 1 (dense early -> select -> gather -> sparse
// middle -> delta scatter -> dense late).  Everything here is host code; every
// step of the computation runs in the kernels it launches.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "../../include/sparse_reslim.h"
#include "kernels.h"

using sr::DType;
using sr::Epi;

namespace sr {
void set_error_message(const std::string& msg);
}  // namespace sr

namespace {

thread_local std::string g_last_msg;

sr_status fail(sr_status st, const char* what) {
  g_last_msg = what;
  return st;
}

// Host-side fault injection for tests of the error paths: the CUDA call with
// index g_fail_at (0-based, counted by g_enqueues since the hook was set) is not
// made and reports cudaErrorLaunchFailure instead.
std::atomic<long long> g_fail_at{-1};
std::atomic<long long> g_enqueues{0};
thread_local bool g_injected = false;

cudaError_t enqueue_gate() {
  const long long n = g_enqueues.fetch_add(1);
  g_injected = n == g_fail_at.load();
  return g_injected ? cudaErrorLaunchFailure : cudaSuccess;
}

sr_status cuda_fail(cudaError_t e, const char* where) {
  g_last_msg = std::string(where) + ": " + cudaGetErrorName(e) + " (" + cudaGetErrorString(e) + ")" +
               (g_injected ? " [injected by sr_debug_fail_enqueue]" : "");
  g_injected = false;
  return SR_ERR_CUDA;
}

// Every CUDA call of the entry points below goes through the injection gate
// first; a failed call returns SR_ERR_CUDA at once, so nothing after it is
// enqueued.
#define SR_CUDA(call, where)                                \
  do {                                                      \
    cudaError_t e__ = enqueue_gate();                       \
    if (e__ == cudaSuccess) e__ = (call);                   \
    if (e__ != cudaSuccess) return cuda_fail(e__, where);   \
  } while (0)

constexpr size_t kAlign = 256;
size_t align_up(size_t v) { return (v + kAlign - 1) / kAlign * kAlign; }

}  // namespace

// Records a message for sr_last_error_message() (used by entry points defined
// in other translation units).
void sr::set_error_message(const std::string& msg) { g_last_msg = msg; }

namespace {
thread_local bool g_pdl = false;
}  // namespace
bool sr::pdl_enabled() { return g_pdl; }
sr::PdlScope::PdlScope(bool on) : prev(g_pdl) { g_pdl = on; }
sr::PdlScope::~PdlScope() { g_pdl = prev; }

namespace {

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

int32_t keep_count(int32_t L, float r) {
  if (L < 1 || !(r > 0.0f) || !(r <= 1.0f)) return -1;
  return static_cast<int32_t>(std::floor(static_cast<double>(r) * static_cast<double>(L)));
}

size_t elem_size(int32_t dtype) { return dtype == SR_BF16 ? 2 : 4; }

// Workspace layout for a config and a maximum routed count Kmax.
struct Plan {
  size_t fault, xs, ln, qkv, att, u, hs, idx, score, splitk, total;
  size_t splitk_floats;   // fp32 split-K scratch of the CUDA-core GEMMs (fp32 storage only)
  size_t block_rows;   // rows the per-block buffers (ln, qkv, att, u) hold
};

Plan make_plan(const sr_config& c, int32_t Kmax) {
  const size_t es = elem_size(c.dtype);
  const size_t rows = size_t(c.B) * c.L;
  const size_t rrows = size_t(c.B) * (Kmax > 0 ? Kmax : 0);
  Plan p{};
  // dense blocks (or the r = 1 path) see all B*L rows; a model that is only a
  // sparse stage, used with keep ratios below 1, sees at most B*Kmax
  p.block_rows = (c.n1 + c.n3 > 0 || Kmax >= c.L) ? rows : rrows;
  const size_t brows = p.block_rows;
  size_t off = 0;
  p.fault = off; off += kAlign;                                   // device fault word
  p.xs = off;    off += align_up(rows * c.D * sizeof(float));     // fp32 residual stream
  p.ln = off;    off += align_up(brows * c.D * es);
  p.qkv = off;   off += align_up(brows * 3 * c.D * es);
  p.att = off;   off += align_up(brows * c.D * es);
  p.u = off;     off += align_up(brows * size_t(c.mlp_hidden) * es);
  p.hs = off;    off += align_up(rrows * c.D * sizeof(float));    // fp32 routed stream
  p.idx = off;   off += align_up(size_t(c.B) * c.L * sizeof(int32_t));
  // top-K scores: one per token, or the FC2 epilogue's partial sums per token
  const int parts = c.dtype == SR_BF16 ? std::max(1, sr::gemm_tc_sqnorm_parts(c.D)) : 1;
  p.score = off; off += align_up(rows * size_t(parts) * sizeof(float));
  // the CUDA-core GEMMs split K in up to 8 slices when their output tiles alone
  // leave SMs idle (the D-wide GEMMs of small row counts)
  p.splitk_floats = c.dtype == SR_F32 ? 8 * brows * size_t(c.D) : 0;
  p.splitk = off; off += align_up(p.splitk_floats * sizeof(float));
  p.total = off;
  return p;
}

sr_status validate_config(const sr_config* c) {
  if (!c) return fail(SR_ERR_INVALID_ARG, "config is NULL");
  if (c->B < 1 || c->L < 1) return fail(SR_ERR_INVALID_ARG, "B and L must be >= 1");
  if (c->heads < 1 || c->D != 64 * c->heads)
    return fail(SR_ERR_UNSUPPORTED, "D must equal 64 * heads (head_dim 64)");
  if (c->mlp_hidden < 64 || c->mlp_hidden % 64 != 0)
    return fail(SR_ERR_UNSUPPORTED, "mlp_hidden must be a positive multiple of 64");
  if (c->n1 < 0 || c->n2 < 0 || c->n3 < 0 || c->n1 + c->n2 + c->n3 < 1)
    return fail(SR_ERR_INVALID_ARG, "block split needs n1, n2, n3 >= 0 and n1 + n2 + n3 >= 1");
  if (c->dtype != SR_F32 && c->dtype != SR_BF16) return fail(SR_ERR_INVALID_ARG, "bad dtype");
  if (c->selector != SR_SEL_RANDOM && c->selector != SR_SEL_TOPK_L2 &&
      c->selector != SR_SEL_LAPLACIAN)
    return fail(SR_ERR_INVALID_ARG, "bad selector");
  if (c->selector == SR_SEL_LAPLACIAN && (c->grid_w < 1 || c->L % c->grid_w != 0))
    return fail(SR_ERR_INVALID_ARG, "the Laplacian selector needs grid_w >= 1 dividing L");
  if (c->shared_indices != 0 && c->shared_indices != 1)
    return fail(SR_ERR_INVALID_ARG, "shared_indices must be 0 or 1");
  if (!(c->ln_eps > 0.0f) || !std::isfinite(c->ln_eps))
    return fail(SR_ERR_INVALID_ARG, "ln_eps must be a positive finite number");
  const int maxD = c->dtype == SR_BF16 ? 2048 : 1024;
  if (c->D > maxD) return fail(SR_ERR_UNSUPPORTED, "D too large for the row kernels");
  if (c->L > sr::select_max_L())
    return fail(SR_ERR_UNSUPPORTED, "L exceeds the selection kernel's shared-memory capacity");
  const double rows = double(c->B) * double(c->L);
  if (rows * double(c->mlp_hidden > 3 * c->D ? c->mlp_hidden : 3 * c->D) >= 2147483647.0)
    return fail(SR_ERR_UNSUPPORTED, "B * L * width exceeds 2^31 elements");
  return SR_OK;
}

}  // namespace

struct TraceRec {
  int kind;
  cudaEvent_t ev0, ev1;
  double flops, bytes;
};

struct sr_handle {
  sr_config cfg;
  DType dt;
  size_t es;
  char* ws;
  size_t ws_bytes;
  int32_t Kmax;
  Plan plan;
  bool trace = false;
  bool fault_cleared = false;   // the fault word is zeroed by the first enqueuing call
  std::vector<TraceRec> pending;
  std::vector<cudaEvent_t> pool;
  sr_trace_entry acc[SR_KERN_COUNT] = {};
  // a batched view of a handle (the implicit ensemble's members as one batch)
  // shares its owner's fault word and trace records
  unsigned int* fault_ptr = nullptr;
  sr_handle* owner = nullptr;
  void* at(size_t off) const { return ws + off; }
  unsigned int* fault() const {
    return fault_ptr ? fault_ptr : static_cast<unsigned int*>(at(plan.fault));
  }
  sr_handle* trace_owner() { return owner ? owner : this; }
  ~sr_handle() {
    for (auto& r : pending) { cudaEventDestroy(r.ev0); cudaEventDestroy(r.ev1); }
    for (auto e : pool) cudaEventDestroy(e);
  }
};

namespace {

cudaEvent_t take_event(sr_handle* h) {
  if (!h->pool.empty()) {
    cudaEvent_t e = h->pool.back();
    h->pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

// Records CUDA events around one launch when the handle traces and the stream
// is not capturing.
struct TraceScope {
  sr_handle* h;
  cudaStream_t s;
  TraceRec rec{};
  bool on = false;
  TraceScope(const sr_handle* hc, int kind, double flops, double bytes, cudaStream_t st)
      : h(const_cast<sr_handle*>(hc)->trace_owner()), s(st) {
    if (!h->trace) return;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(s, &cs) != cudaSuccess || cs != cudaStreamCaptureStatusNone) return;
    rec.kind = kind; rec.flops = flops; rec.bytes = bytes;
    rec.ev0 = take_event(h); rec.ev1 = take_event(h);
    if (!rec.ev0 || !rec.ev1) return;
    on = cudaEventRecord(rec.ev0, s) == cudaSuccess;
  }
  ~TraceScope() {
    if (on && cudaEventRecord(rec.ev1, s) == cudaSuccess) h->pending.push_back(rec);
  }
};

// GEMM and attention dispatch by dtype.
cudaError_t gemm(const sr_handle* h, Epi epi, const void* A, const void* W, int M, int N, int K,
                 const sr::EpiArgs& ea, cudaStream_t s) {
  if (h->dt == DType::BF16) return sr::launch_gemm_tc(epi, A, W, M, N, K, ea, s);
  return sr::launch_gemm_simt(h->dt, epi, A, W, M, N, K, ea, s,
                              static_cast<float*>(h->at(h->plan.splitk)), h->plan.splitk_floats);
}

cudaError_t attention(const sr_handle* h, const void* qkv, void* out, int B, int T,
                      cudaStream_t s) {
  if (h->dt == DType::BF16) return sr::launch_attention_tc(qkv, out, B, T, h->cfg.heads, h->fault(), s);
  return sr::launch_attention_simt(h->dt, qkv, out, B, T, h->cfg.heads, s);
}

// One pre-LN block (Sec. 3.3 Eq. 11) on the fp32 residual stream x [B*T, D], in
// place.  With `sqnorm` set, the FC2 epilogue also writes each row's squared
// norm (values rounded to the storage dtype) as partial sums per half tile to
// sqnorm [B*T][parts], the scores of the top-K selector.  With `scatter` set this is the last sparse block: its FC2 epilogue
// writes x0 + (h_out - h0) into the rows idx of the stream `scatter_out`
// [B*Lx, D] instead of x.  With `gather_from` set this is the first sparse
// block: its LN1 reads the rows idx of the stream `gather_from` [B*Lx, D]
// directly and also writes them to x (the gather of Eq. 8, fused).
sr_status run_block(const sr_handle* hd, float* x, int B, int T, const sr_block_weights& w,
                    bool scatter, float* scatter_out, const int32_t* idx, int Lx,
                    cudaStream_t s, const float* gather_from = nullptr, float* sqnorm = nullptr) {
  const sr_config& c = hd->cfg;
  const int rows = B * T, D = c.D, H = c.mlp_hidden;
  const double es = double(hd->es), R = double(rows);
  void* ln = hd->at(hd->plan.ln);
  void* qkv = hd->at(hd->plan.qkv);
  void* att = hd->at(hd->plan.att);
  void* u = hd->at(hd->plan.u);
  const double ln_bytes = R * D * (4.0 + es) + 2.0 * D * es;
  if (gather_from) {
    // reads the selected rows, writes LN1 and the fp32 copy h0, plus the index set
    TraceScope t(hd, SR_KERN_GATHER, 0.0, R * D * (8.0 + es) + 4.0 * R + 2.0 * D * es, s);
    SR_CUDA(sr::launch_layernorm(hd->dt, gather_from, w.ln1_g, w.ln1_b, ln, rows, D, c.ln_eps, s,
                                 idx, Lx, T, x),
            "gather + layernorm1");
  } else {
    TraceScope t(hd, SR_KERN_LAYERNORM, 0.0, ln_bytes, s);
    SR_CUDA(sr::launch_layernorm(hd->dt, x, w.ln1_g, w.ln1_b, ln, rows, D, c.ln_eps, s), "layernorm1");
  }
  {
    TraceScope t(hd, SR_KERN_GEMM_QKV, 2.0 * R * 3 * D * D,
                 (R * D + 3.0 * D * D + R * 3 * D + 3.0 * D) * es, s);
    sr::EpiArgs e1{w.bqkv, nullptr, qkv, nullptr, 0, 0, hd->fault()};
    SR_CUDA(gemm(hd, Epi::Bias, ln, w.wqkv, rows, 3 * D, D, e1, s), "qkv gemm");
  }
  {
    TraceScope t(hd, SR_KERN_ATTENTION, 4.0 * B * c.heads * double(T) * T * 64.0,
                 (R * 3 * D + R * D) * es, s);
    SR_CUDA(attention(hd, qkv, att, B, T, s), "attention");
  }
  {
    TraceScope t(hd, SR_KERN_GEMM_OUT, 2.0 * R * D * D, (R * D + 1.0 * D * D + D) * es + 8.0 * R * D, s);
    sr::EpiArgs e2{w.bo, x, x, nullptr, 0, 0, hd->fault()};
    SR_CUDA(gemm(hd, Epi::BiasResidual, att, w.wo, rows, D, D, e2, s), "out-proj gemm");
  }
  {
    TraceScope t(hd, SR_KERN_LAYERNORM, 0.0, ln_bytes, s);
    SR_CUDA(sr::launch_layernorm(hd->dt, x, w.ln2_g, w.ln2_b, ln, rows, D, c.ln_eps, s), "layernorm2");
  }
  {
    TraceScope t(hd, SR_KERN_GEMM_FC1, 2.0 * R * H * D, (R * D + 1.0 * H * D + R * H + H) * es, s);
    sr::EpiArgs e3{w.b1, nullptr, u, nullptr, 0, 0, hd->fault()};
    SR_CUDA(gemm(hd, Epi::BiasGelu, ln, w.w1, rows, H, D, e3, s), "fc1 gemm");
  }
  if (!scatter) {
    TraceScope t(hd, SR_KERN_GEMM_FC2, 2.0 * R * D * H, (R * H + 1.0 * D * H + D) * es + 8.0 * R * D, s);
    sr::EpiArgs e4{w.b2, x, x, nullptr, 0, 0, hd->fault(), sqnorm};
    SR_CUDA(gemm(hd, Epi::BiasResidual, u, w.w2, rows, D, H, e4, s), "fc2 gemm");
  } else {
    // reads h and x0 rows, writes the scattered rows, plus the index set
    TraceScope t(hd, SR_KERN_GEMM_FC2_SCATTER, 2.0 * R * D * H,
                 (R * H + 1.0 * D * H + D) * es + 12.0 * R * D + 4.0 * R, s);
    sr::EpiArgs e4{w.b2, x, scatter_out, idx, T, Lx, hd->fault()};
    SR_CUDA(gemm(hd, Epi::BiasResidualScatter, u, w.w2, rows, D, H, e4, s), "fc2 scatter gemm");
  }
  return SR_OK;
}

bool weights_ok(const sr_block_weights& w) {
  const void* p[12] = {w.ln1_g, w.ln1_b, w.wqkv, w.bqkv, w.wo, w.bo,
                       w.ln2_g, w.ln2_b, w.w1, w.b1, w.w2, w.b2};
  for (const void* q : p)
    if (!q || !aligned(q, 16)) return false;
  return true;
}

// Whether sr_forward takes the top-K scores from the last dense-early block's FC2
// epilogue instead of a pass over the stream (the GEMM must be a tcgen05 pair
// GEMM with the TMA residual epilogue).
bool scores_fused(const sr_handle* h) {
  const sr_config& c = h->cfg;
  return c.selector == SR_SEL_TOPK_L2 && h->dt == DType::BF16 && c.n1 > 0 &&
         sr::gemm_tc_sqnorm_parts(c.D) > 0;
}

// score_ready: the top-K scores are already in the workspace (fused into FC2)
sr_status do_select(sr_handle* h, const float* x, int32_t K, uint64_t seed, int32_t* idx,
                    cudaStream_t s, bool score_ready = false) {
  const sr_config& c = h->cfg;
  const bool norms = c.selector == SR_SEL_TOPK_L2 && !score_ready;
  const bool lap = c.selector == SR_SEL_LAPLACIAN;
  // the Laplacian reads every token once (its four neighbours come from L2)
  const double sel_bytes = 4.0 * c.B * K +
      (c.selector != SR_SEL_RANDOM ? 4.0 * c.B * c.L : 0.0) +
      (norms || lap ? double(c.B) * c.L * c.D * 4.0 : 0.0);
  TraceScope t(h, SR_KERN_SELECT, 0.0, sel_bytes, s);
  if (c.selector == SR_SEL_RANDOM) {
    SR_CUDA(sr::launch_select_random(c.B, c.L, K, seed, c.shared_indices, idx, s), "select_random");
  } else {
    float* score = static_cast<float*>(h->at(h->plan.score));
    if (norms) SR_CUDA(sr::launch_token_sq_norms(h->dt, x, c.B * c.L, c.D, score, s), "token norms");
    if (lap)
      SR_CUDA(sr::launch_token_laplacian(h->dt, x, c.B, c.L, c.grid_w, c.D, score, s),
              "token Laplacian scores");
    const int parts = norms || lap ? 1 : sr::gemm_tc_sqnorm_parts(c.D);
    SR_CUDA(sr::launch_select_topk(c.B, c.L, K, score, idx, s, parts), "select_topk");
  }
  return SR_OK;
}

}  // namespace

extern "C" {

int32_t sr_keep_count(int32_t L, float keep_ratio) { return keep_count(L, keep_ratio); }

size_t sr_workspace_bytes(const sr_config* cfg, float max_keep_ratio) {
  if (validate_config(cfg) != SR_OK) return 0;
  const int32_t K = keep_count(cfg->L, max_keep_ratio);
  if (K < 0) return 0;
  return make_plan(*cfg, K).total;
}

sr_status sr_create(const sr_config* cfg, void* workspace, size_t ws_bytes, sr_handle** out) {
  if (!out) return fail(SR_ERR_INVALID_ARG, "out handle pointer is NULL");
  *out = nullptr;
  sr_status st = validate_config(cfg);
  if (st != SR_OK) return st;
  if (!workspace || !aligned(workspace, kAlign))
    return fail(SR_ERR_WORKSPACE, "workspace is NULL or not 256-byte aligned");
  // the largest Kmax whose plan fits: the routed buffers scale with Kmax
  const Plan full = make_plan(*cfg, cfg->L);
  int32_t Kmax = cfg->L;
  if (ws_bytes < full.total) {
    const Plan none = make_plan(*cfg, 0);
    if (ws_bytes < none.total) return fail(SR_ERR_WORKSPACE, "workspace too small");
    const size_t per_row = size_t(cfg->B) * cfg->D * sizeof(float);
    Kmax = int32_t((ws_bytes - none.total) / (per_row ? per_row : 1));
    while (Kmax > 0 && make_plan(*cfg, Kmax).total > ws_bytes) --Kmax;
    if (Kmax < 1) return fail(SR_ERR_WORKSPACE, "workspace too small for any routed token");
  }
  sr_handle* h = new (std::nothrow) sr_handle;
  if (!h) return fail(SR_ERR_INTERNAL, "host allocation failed");
  h->cfg = *cfg;
  h->dt = cfg->dtype == SR_BF16 ? DType::BF16 : DType::F32;
  h->es = elem_size(cfg->dtype);
  h->ws = static_cast<char*>(workspace);
  h->ws_bytes = ws_bytes;
  h->Kmax = Kmax;
  h->plan = make_plan(*cfg, Kmax);
  *out = h;
  return SR_OK;
}

sr_status sr_destroy(sr_handle* h) {
  delete h;
  return SR_OK;
}

sr_status sr_select(sr_handle* h, const void* x, float keep_ratio, uint64_t seed, int32_t* idx,
                    int32_t* K_out, void* stream) {
  if (!h) return fail(SR_ERR_INVALID_ARG, "handle is NULL");
  const int32_t K = keep_count(h->cfg.L, keep_ratio);
  if (K < 0) return fail(SR_ERR_INVALID_ARG, "keep_ratio must lie in (0, 1]");
  if (K < 1) return fail(SR_ERR_INVALID_ARG, "K = floor(L * keep_ratio) is 0");
  if (!idx || !aligned(idx, 4)) return fail(SR_ERR_INVALID_ARG, "idx is NULL or misaligned");
  if (h->cfg.selector != SR_SEL_RANDOM && (!x || !aligned(x, 16)))
    return fail(SR_ERR_INVALID_ARG, "score-based selection needs a 16-byte aligned x");
  if (K_out) *K_out = K;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  float* xs = nullptr;
  if (h->cfg.selector != SR_SEL_RANDOM) {
    // the scores are taken of the stored activations: widen them into the stream buffer
    xs = static_cast<float*>(h->at(h->plan.xs));
    SR_CUDA(sr::launch_widen(h->dt, x, xs, size_t(h->cfg.B) * h->cfg.L * h->cfg.D, s), "widen x");
  }
  return do_select(h, xs, K, seed, idx, s);
}

namespace {

// Host checks shared by sr_forward and sr_forward_ensemble (no CUDA calls).
sr_status check_forward_args(const sr_handle* h, const void* x, const sr_block_weights* w,
                             float keep_ratio, const void* out, int32_t* K) {
  if (!h) return fail(SR_ERR_INVALID_ARG, "handle is NULL");
  const sr_config& c = h->cfg;
  const int N = c.n1 + c.n2 + c.n3;
  if (!x || !out || !aligned(x, 16) || !aligned(out, 16))
    return fail(SR_ERR_INVALID_ARG, "x and out must be non-NULL and 16-byte aligned");
  if (!w) return fail(SR_ERR_INVALID_ARG, "weights array is NULL");
  for (int i = 0; i < N; ++i)
    if (!weights_ok(w[i])) return fail(SR_ERR_INVALID_ARG, "a block weight pointer is NULL or misaligned");
  *K = keep_count(c.L, keep_ratio);
  if (*K < 0) return fail(SR_ERR_INVALID_ARG, "keep_ratio must lie in (0, 1]");
  const bool route = keep_ratio < 1.0f && c.n2 > 0;
  if (*K < 1 && route) return fail(SR_ERR_INVALID_ARG, "K = floor(L * keep_ratio) is 0");
  if (route && *K > h->Kmax) return fail(SR_ERR_WORKSPACE, "K exceeds the workspace's routed capacity");
  if (!route && c.n2 > 0 && size_t(c.B) * c.L > h->plan.block_rows)
    return fail(SR_ERR_WORKSPACE, "workspace sized for keep ratios below 1 only");
  const size_t bytes = size_t(c.B) * c.L * c.D * h->es;
  const char* xb = static_cast<const char*>(x);
  const char* ob = static_cast<const char*>(out);
  if (xb != ob && xb < ob + bytes && ob < xb + bytes)
    return fail(SR_ERR_INVALID_ARG, "out partially overlaps x");
  return SR_OK;
}

// x (storage dtype) into the fp32 stream xs, then the n1 dense-early blocks.
sr_status widen_and_early(sr_handle* h, const void* x, const sr_block_weights* w, float* xs,
                          cudaStream_t s) {
  const sr_config& c = h->cfg;
  if (!h->fault_cleared) {
    SR_CUDA(cudaMemsetAsync(h->fault(), 0, sizeof(unsigned int), s), "clear fault word");
    h->fault_cleared = true;
  }
  const size_t n = size_t(c.B) * c.L * c.D;
  // the top-K scores come out of the last dense-early block's FC2 epilogue as
  // partial sums per row
  float* score = scores_fused(h) ? static_cast<float*>(h->at(h->plan.score)) : nullptr;
  {
    // the residual stream is held in fp32 for the whole forward
    TraceScope t(h, SR_KERN_COPY, 0.0, double(n) * (h->es + 4.0), s);
    SR_CUDA(sr::launch_widen(h->dt, x, xs, n, s), "widen x");
  }
  // every later kernel may start while its predecessor finishes (not while
  // tracing, which records events between kernels)
  const sr::PdlScope pdl(!h->trace);
  sr_status st;
  for (int i = 0; i < c.n1; ++i)
    if ((st = run_block(h, xs, c.B, c.L, w[i], false, nullptr, nullptr, 0, s, nullptr,
                        i == c.n1 - 1 ? score : nullptr)) != SR_OK)
      return st;
  return SR_OK;
}

// The sparse middle (gather fused into its first LN1, delta scatter into its
// last FC2) and the dense-late blocks, in place on the fp32 stream xs of h,
// given the index set idx [B, K] (Alg. 1 after the selection).  With route false
// the middle blocks run densely (r = 1, or no sparse blocks).
sr_status blocks_after_select(sr_handle* h, float* xs, const sr_block_weights* w, bool route,
                              int32_t K, const int32_t* idx, cudaStream_t s) {
  const sr_config& c = h->cfg;
  const int N = c.n1 + c.n2 + c.n3;
  sr_status st;
  if (route) {
    float* hs = static_cast<float*>(h->at(h->plan.hs));
    for (int i = c.n1; i < c.n1 + c.n2; ++i) {
      const bool last = i == c.n1 + c.n2 - 1;
      if ((st = run_block(h, hs, c.B, K, w[i], last, xs, idx, c.L, s, i == c.n1 ? xs : nullptr)) !=
          SR_OK)
        return st;
    }
  } else {
    for (int i = c.n1; i < c.n1 + c.n2; ++i)
      if ((st = run_block(h, xs, c.B, c.L, w[i], false, nullptr, nullptr, 0, s)) != SR_OK) return st;
  }
  for (int i = c.n1 + c.n2; i < N; ++i)
    if ((st = run_block(h, xs, c.B, c.L, w[i], false, nullptr, nullptr, 0, s)) != SR_OK) return st;
  return SR_OK;
}

// Everything after the dense-early blocks, in place on the fp32 stream xs:
// selection, gather, the sparse middle with the delta scatter fused into its
// last block, and the dense-late blocks (Alg. 1 after its dense-early loop).
sr_status route_and_late(sr_handle* h, float* xs, const sr_block_weights* w, float keep_ratio,
                         int32_t K, uint64_t seed, int32_t* idx_out, cudaStream_t s) {
  const sr_config& c = h->cfg;
  const bool route = keep_ratio < 1.0f && c.n2 > 0;
  sr_status st;
  int32_t* idx = idx_out ? idx_out : static_cast<int32_t*>(h->at(h->plan.idx));
  if (route || idx_out)
    if ((st = do_select(h, xs, K, seed, idx, s, scores_fused(h))) != SR_OK) return st;
  return blocks_after_select(h, xs, w, route, K, idx, s);
}

// The config of M members of the implicit ensemble run as one batch of M * B
// samples (member m's sample b is sample m * B + b).
sr_config ensemble_batch_config(const sr_config& c, int32_t M) {
  sr_config e = c;
  e.B = c.B * M;
  return e;
}

}  // namespace

sr_status sr_forward(sr_handle* h, const void* x, const sr_block_weights* w, float keep_ratio,
                     uint64_t seed, void* out, int32_t* idx_out, void* stream) {
  int32_t K = 0;
  sr_status st = check_forward_args(h, x, w, keep_ratio, out, &K);
  if (st != SR_OK) return st;
  if (idx_out && !aligned(idx_out, 4)) return fail(SR_ERR_INVALID_ARG, "idx_out misaligned");
  if (idx_out && K < 1) return fail(SR_ERR_INVALID_ARG, "K = floor(L * keep_ratio) is 0");
  const sr_config& c = h->cfg;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t n = size_t(c.B) * c.L * c.D;
  float* xs = static_cast<float*>(h->at(h->plan.xs));
  const sr::PdlScope pdl(false);             // the widen waits for whatever came before
  if ((st = widen_and_early(h, x, w, xs, s)) != SR_OK) return st;
  const sr::PdlScope pdl_rest(!h->trace);
  if ((st = route_and_late(h, xs, w, keep_ratio, K, seed, idx_out, s)) != SR_OK) return st;
  {
    TraceScope t(h, SR_KERN_COPY, 0.0, double(n) * (h->es + 4.0), s);
    SR_CUDA(sr::launch_narrow(h->dt, xs, out, n, s), "narrow out");
  }
  return SR_OK;
}

size_t sr_ensemble_workspace_bytes(const sr_config* cfg, int32_t M, float max_keep_ratio) {
  if (validate_config(cfg) != SR_OK || M < 1) return 0;
  if (double(cfg->B) * M > 2147483647.0) return 0;
  const int32_t K = keep_count(cfg->L, max_keep_ratio);
  if (K < 0) return 0;
  const sr_config e = ensemble_batch_config(*cfg, M);
  if (validate_config(&e) != SR_OK) return 0;
  return make_plan(e, K).total;
}

sr_status sr_forward_ensemble(sr_handle* h, const void* x, const sr_block_weights* w,
                              float keep_ratio, const uint64_t* seeds, int32_t M,
                              void* ens_workspace, size_t ens_ws_bytes, void* out,
                              void* members_out, int32_t* idx_out, void* stream) {
  int32_t K = 0;
  sr_status st = check_forward_args(h, x, w, keep_ratio, out, &K);
  if (st != SR_OK) return st;
  if (M < 1 || !seeds) return fail(SR_ERR_INVALID_ARG, "need M >= 1 seeds");
  const sr_config& c = h->cfg;
  const size_t n = size_t(c.B) * c.L * c.D;
  if (double(c.B) * M > 2147483647.0) return fail(SR_ERR_UNSUPPORTED, "B * M too large");
  const sr_config ec = ensemble_batch_config(c, M);
  if ((st = validate_config(&ec)) != SR_OK) return st;
  const Plan ep = make_plan(ec, K > 0 ? K : 0);
  if (!ens_workspace || !aligned(ens_workspace, kAlign) || ens_ws_bytes < ep.total)
    return fail(SR_ERR_WORKSPACE, "ensemble workspace NULL, misaligned or too small");
  if (members_out && !aligned(members_out, 16))
    return fail(SR_ERR_INVALID_ARG, "members_out must be 16-byte aligned");
  if (idx_out && (!aligned(idx_out, 4) || K < 1))
    return fail(SR_ERR_INVALID_ARG, "idx_out misaligned or K = 0");
  const size_t bytes = n * h->es;
  if (members_out) {
    // members_out must not overlap x or out
    const char* mb = static_cast<const char*>(members_out);
    const char* xb = static_cast<const char*>(x);
    const char* ob = static_cast<const char*>(out);
    const size_t mbytes = size_t(M) * bytes;
    if ((mb < xb + bytes && xb < mb + mbytes) || (mb < ob + bytes && ob < mb + mbytes))
      return fail(SR_ERR_INVALID_ARG, "members_out overlaps x or out");
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  float* xs = static_cast<float*>(h->at(h->plan.xs));
  const sr::PdlScope pdl(false);
  // the dense-early blocks do not depend on the seed: once for all members
  if ((st = widen_and_early(h, x, w, xs, s)) != SR_OK) return st;
  const sr::PdlScope pdl_rest(!h->trace);
  const bool route = keep_ratio < 1.0f && c.n2 > 0;
  if (!route) {
    // nothing is routed: every member is the same dense forward, and so is
    // their mean
    for (int32_t m = 0; idx_out && m < M; ++m)
      if ((st = do_select(h, xs, K, seeds[m], idx_out + size_t(m) * c.B * K, s, scores_fused(h))) !=
          SR_OK)
        return st;
    if ((st = blocks_after_select(h, xs, w, false, K, nullptr, s)) != SR_OK) return st;
    TraceScope t(h, SR_KERN_COPY, 0.0, double(n) * (h->es + 4.0) * (1 + (members_out ? M : 0)), s);
    for (int32_t m = 0; members_out && m < M; ++m)
      SR_CUDA(sr::launch_narrow(h->dt, xs, static_cast<char*>(members_out) + size_t(m) * bytes, n, s),
              "narrow member");
    SR_CUDA(sr::launch_narrow(h->dt, xs, out, n, s), "narrow out");
    return SR_OK;
  }
  // the M members run as one batch of M * B samples on a view of the handle
  // over the ensemble workspace; each member's index set is selected from the
  // shared dense-early result with its own seed, exactly as sr_forward does
  sr_handle v;
  v.cfg = ec;
  v.dt = h->dt;
  v.es = h->es;
  v.ws = static_cast<char*>(ens_workspace);
  v.ws_bytes = ens_ws_bytes;
  v.Kmax = K;
  v.plan = ep;
  v.trace = h->trace;
  v.fault_ptr = h->fault();
  v.owner = h;
  float* xe = static_cast<float*>(v.at(ep.xs));
  int32_t* idx = idx_out ? idx_out : static_cast<int32_t*>(v.at(ep.idx));
  for (int32_t m = 0; m < M; ++m)
    if ((st = do_select(h, xs, K, seeds[m], idx + size_t(m) * c.B * K, s, scores_fused(h))) != SR_OK)
      return st;
  {
    TraceScope t(h, SR_KERN_COPY, 0.0, 4.0 * double(n) * (1 + M), s);
    SR_CUDA(sr::launch_replicate(xs, xe, n, M, s), "replicate the dense-early result");
  }
  if ((st = blocks_after_select(&v, xe, w, true, K, idx, s)) != SR_OK) return st;
  if (members_out) {
    TraceScope t(h, SR_KERN_COPY, 0.0, double(M) * n * (h->es + 4.0), s);
    SR_CUDA(sr::launch_narrow(h->dt, xe, members_out, size_t(M) * n, s), "narrow members");
  }
  {
    // the mean of the members' fp32 results (summed in member order), rounded once
    TraceScope t(h, SR_KERN_COPY, 0.0, double(n) * (4.0 * M + h->es), s);
    SR_CUDA(sr::launch_mean_narrow(h->dt, xe, M, n, 1.0f / float(M), out, s), "narrow mean");
  }
  return SR_OK;
}

sr_status sr_cross_attention(const void* q, const void* kv, int32_t B, int32_t Tq, int32_t Tkv,
                             int32_t heads, void* out, uint32_t* fault, void* stream) {
  if (!q || !kv || !out || !aligned(q, 16) || !aligned(kv, 16) || !aligned(out, 16))
    return fail(SR_ERR_INVALID_ARG, "q, kv and out must be non-NULL and 16-byte aligned");
  if (fault && !aligned(fault, 4)) return fail(SR_ERR_INVALID_ARG, "fault word misaligned");
  if (B < 1 || Tq < 1 || Tkv < 1) return fail(SR_ERR_INVALID_ARG, "B, Tq and Tkv must be >= 1");
  if (heads < 1 || heads > 32) return fail(SR_ERR_UNSUPPORTED, "heads must lie in 1..32");
  const double D = 64.0 * heads;
  if (double(B) * Tq * D >= 2147483647.0 || double(B) * Tkv * 2.0 * D >= 2147483647.0)
    return fail(SR_ERR_UNSUPPORTED, "B * T * width exceeds 2^31 elements");
  const size_t qbytes = size_t(B) * Tq * size_t(D) * 2, kvbytes = size_t(B) * Tkv * size_t(D) * 4;
  const char* ob = static_cast<const char*>(out);
  const char* qb = static_cast<const char*>(q);
  const char* kb = static_cast<const char*>(kv);
  if ((ob < qb + qbytes && qb < ob + qbytes) || (ob < kb + kvbytes && kb < ob + qbytes))
    return fail(SR_ERR_INVALID_ARG, "out overlaps q or kv");
  SR_CUDA(sr::launch_cross_attention_tc(q, kv, out, B, Tq, Tkv, heads, fault,
                                        static_cast<cudaStream_t>(stream)),
          "cross attention");
  return SR_OK;
}

sr_status sr_forward_host(sr_handle* h, const void* x_host, const sr_block_weights* w,
                          float keep_ratio, uint64_t seed, void* dev_xout, void* out_host,
                          int32_t* idx_out, void* stream) {
  if (!h) return fail(SR_ERR_INVALID_ARG, "handle is NULL");
  if (!x_host || !out_host || !dev_xout)
    return fail(SR_ERR_INVALID_ARG, "x_host, dev_xout and out_host must be non-NULL");
  // every argument is checked before the first copy is enqueued
  int32_t K = 0;
  sr_status st = check_forward_args(h, dev_xout, w, keep_ratio, dev_xout, &K);
  if (st != SR_OK) return st;
  if (idx_out && !aligned(idx_out, 4)) return fail(SR_ERR_INVALID_ARG, "idx_out misaligned");
  if (idx_out && K < 1) return fail(SR_ERR_INVALID_ARG, "K = floor(L * keep_ratio) is 0");
  const sr_config& c = h->cfg;
  const size_t bytes = size_t(c.B) * c.L * c.D * h->es;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  SR_CUDA(cudaMemcpyAsync(dev_xout, x_host, bytes, cudaMemcpyHostToDevice, s), "copy x host -> device");
  st = sr_forward(h, dev_xout, w, keep_ratio, seed, dev_xout, idx_out, stream);
  if (st != SR_OK) return st;
  SR_CUDA(cudaMemcpyAsync(out_host, dev_xout, bytes, cudaMemcpyDeviceToHost, s), "copy out device -> host");
  return SR_OK;
}

sr_status sr_trace_enable(sr_handle* h, int enable) {
  if (!h) return fail(SR_ERR_INVALID_ARG, "handle is NULL");
  h->trace = enable != 0;
  return SR_OK;
}

sr_status sr_trace_read(sr_handle* h, sr_trace_entry* out, int reset) {
  if (!h) return fail(SR_ERR_INVALID_ARG, "handle is NULL");
  for (auto& r : h->pending) {
    SR_CUDA(cudaEventSynchronize(r.ev1), "trace event sync");
    float ms = 0.f;
    SR_CUDA(cudaEventElapsedTime(&ms, r.ev0, r.ev1), "trace elapsed time");
    sr_trace_entry& a = h->acc[r.kind];
    a.ms += ms; a.launches += 1; a.flops += r.flops; a.bytes += r.bytes;
    h->pool.push_back(r.ev0);
    h->pool.push_back(r.ev1);
  }
  h->pending.clear();
  if (out)
    for (int k = 0; k < SR_KERN_COUNT; ++k) out[k] = h->acc[k];
  if (reset)
    for (int k = 0; k < SR_KERN_COUNT; ++k) h->acc[k] = sr_trace_entry{};
  return SR_OK;
}

const char* sr_status_string(sr_status s) {
  switch (s) {
    case SR_OK: return "SR_OK";
    case SR_ERR_INVALID_ARG: return "SR_ERR_INVALID_ARG: invalid argument";
    case SR_ERR_UNSUPPORTED: return "SR_ERR_UNSUPPORTED: configuration not supported";
    case SR_ERR_WORKSPACE: return "SR_ERR_WORKSPACE: workspace missing or too small";
    case SR_ERR_CUDA: return "SR_ERR_CUDA: CUDA call failed";
    case SR_ERR_INTERNAL: return "SR_ERR_INTERNAL: internal error";
  }
  return "unknown sr_status";
}

const char* sr_last_error_message(void) { return g_last_msg.c_str(); }

void sr_debug_fail_enqueue(int64_t n) {
  g_enqueues.store(0);
  g_fail_at.store(n < 0 ? -1 : static_cast<long long>(n));
}

int64_t sr_debug_enqueue_count(void) { return static_cast<int64_t>(g_enqueues.load()); }

sr_status sr_device_fault(sr_handle* h, uint32_t* fault, int clear, void* stream) {
  if (!h || !fault) return fail(SR_ERR_INVALID_ARG, "handle or fault is NULL");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unsigned int f = 0;
  SR_CUDA(cudaMemcpyAsync(&f, h->fault(), sizeof(f), cudaMemcpyDeviceToHost, s), "read fault word");
  SR_CUDA(cudaStreamSynchronize(s), "stream synchronize");
  if (clear) SR_CUDA(cudaMemsetAsync(h->fault(), 0, sizeof(f), s), "clear fault word");
  *fault = f;
  return SR_OK;
}

}  // extern "C"
