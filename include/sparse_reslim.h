/*
 * sparse_reslim.h -- C ABI of the GB300 (sm_103a) Sparse-Reslim encoder forward.
 *
 * Sparse-Reslim (arxiv 2607.02829) splits the N pre-LN ViT blocks of a
 * weather-forecasting encoder into n1 dense-early, n2 sparse-middle and n3
 * dense-late blocks (Sec. 3.2, Eq. 7).  Between the first two stages K =
 * floor(L * r) tokens per sample are selected (Sec. 3.2), gathered and run
 * through the middle blocks (Eq. 8); the residual delta h - h0 is scattered back
 * so that unselected tokens keep their pre-routing values exactly (Eq. 9); the
 * closing dense blocks then run on all L tokens (Alg. 1).
 *
 * Conventions shared by every call:
 *  - All tensors are dense, row-major and live in device memory owned by the
 *    caller, unless a parameter says "host".  The library never allocates
 *    device memory on these calls; scratch space is the caller's workspace.
 *  - Element type is the config's dtype (fp32 or bf16) for activations and
 *    all block weights, including LayerNorm parameters and biases.  Index
 *    sets are int32.
 *  - Every call is stream-ordered and asynchronous on `stream` (a
 *    cudaStream_t; NULL means the legacy default stream) and returns after
 *    enqueueing work.  Arguments are validated on the host before any launch;
 *    an invalid call enqueues nothing.
 *  - Errors are return codes (sr_status); nothing is thrown and nothing exits.
 *    A CUDA error reported by a launch or an asynchronous copy maps to
 *    SR_ERR_CUDA; the failing CUDA call's message is kept per thread and
 *    returned by sr_last_error_message().
 */
#ifndef SPARSE_RESLIM_H
#define SPARSE_RESLIM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SR_OK = 0,
  SR_ERR_INVALID_ARG = 1,   /* a pointer, size, ratio or config field is invalid */
  SR_ERR_UNSUPPORTED = 2,   /* valid for the method, not supported by these kernels */
  SR_ERR_WORKSPACE = 3,     /* workspace missing, misaligned or too small */
  SR_ERR_CUDA = 4,          /* a CUDA runtime call or kernel launch failed */
  SR_ERR_INTERNAL = 5
} sr_status;

typedef enum { SR_F32 = 0, SR_BF16 = 1 } sr_dtype;

/* Token selector at the dense-early / sparse-middle boundary.
 *  SR_SEL_RANDOM : K tokens uniformly without replacement, sorted ascending
 *                  (Sec. 3.2).  The draw is defined by SplitMix64 keys
 *                  (Steele, Lea & Flood 2014): key(b,i) = mix64(seed +
 *                  0x9E3779B97F4A7C15 * (1 + b' * L + i)), b' = b, or 0 when
 *                  shared_indices; the K smallest (key, i) pairs are kept.
 *  SR_SEL_TOPK_L2: the K tokens with the largest L2 norm of the last
 *                  dense-early block's output (the activation-norm selector of
 *                  App. B.2, Table 11); ties go to the lower token index.  The
 *                  squared norm of the stored activations (each value rounded
 *                  to the storage dtype) is accumulated in fp32.  In
 *                  sr_forward with bf16 storage, n1 >= 1 and D % 128 == 0 the
 *                  norms come out of the last dense-early block's FC2
 *                  epilogue; otherwise (and always in sr_select) a separate
 *                  pass reads the stream.
 *  SR_SEL_LAPLACIAN: the K tokens with the largest Laplacian score of the
 *                  last dense-early block's output (the gradient-based
 *                  sampler of App. B.2, Table 11, which gives no formula; this
 *                  library reads it as follows).  Tokens lie row-major on the
 *                  patch grid, grid_w per latitude row; the score of token
 *                  (i, j) is the squared L2 norm over D of the 5-point
 *                  Laplacian x(i-1,j) + x(i+1,j) + x(i,j-1) + x(i,j+1) -
 *                  4 x(i,j), with longitude periodic and the first and last
 *                  latitude rows reflected onto themselves (x(-1,j) = x(0,j),
 *                  x(H,j) = x(H-1,j)).  Values are rounded to the storage
 *                  dtype first and the score is accumulated in fp32; ties go
 *                  to the lower token index. */
typedef enum { SR_SEL_RANDOM = 0, SR_SEL_TOPK_L2 = 1, SR_SEL_LAPLACIAN = 2 } sr_selector;

typedef struct {
  int32_t B;              /* batch size, >= 1 */
  int32_t L;              /* tokens per sample, >= 1 */
  int32_t D;              /* model width; D == 64 * heads (head_dim 64); D % 64 == 0 */
  int32_t heads;          /* attention heads, >= 1 */
  int32_t mlp_hidden;     /* MLP hidden width (4 * D in the paper's blocks); % 64 == 0 */
  int32_t n1, n2, n3;     /* block split, Sec. 3.2 Eq. 7; each >= 0, n1 + n2 + n3 >= 1 */
  int32_t dtype;          /* sr_dtype */
  int32_t selector;       /* sr_selector */
  int32_t shared_indices; /* 0: one index set per sample (Sec. 3.2 text);
                             1: one set for the whole batch (App. A.4 listing) */
  float ln_eps;           /* LayerNorm epsilon, > 0 (PyTorch's default is 1e-5) */
  int32_t grid_w;         /* tokens per latitude row of the patch grid; L % grid_w == 0.
                             Read by SR_SEL_LAPLACIAN only (0 otherwise) */
} sr_config;

/* Device pointers of one pre-LN block (Sec. 3.3 Eq. 11), nn.Linear layout
 * ([out_features, in_features], row-major):
 *   ln1_g, ln1_b [D]; wqkv [3D, D] (rows [0,D) = q, [D,2D) = k, [2D,3D) = v,
 *   head h owning rows [64h, 64h+64) of each); bqkv [3D]; wo [D, D]; bo [D];
 *   ln2_g, ln2_b [D]; w1 [H, D]; b1 [H]; w2 [D, H]; b2 [D]   (H = mlp_hidden).
 * Every pointer must be non-NULL and 16-byte aligned. */
typedef struct {
  const void *ln1_g, *ln1_b, *wqkv, *bqkv, *wo, *bo;
  const void *ln2_g, *ln2_b, *w1, *b1, *w2, *b2;
} sr_block_weights;

typedef struct sr_handle sr_handle;

/* K = floor(L * keep_ratio) (Sec. 3.2; App. A.4 writes int(r * L)): the
 * product is formed in double precision and truncated.  Returns -1 when
 * keep_ratio is outside (0, 1] or L < 1. */
int32_t sr_keep_count(int32_t L, float keep_ratio);

/* Bytes of device workspace sr_create needs for `cfg` when every later call
 * uses keep_ratio <= max_keep_ratio.  Returns 0 for an invalid config. */
size_t sr_workspace_bytes(const sr_config* cfg, float max_keep_ratio);

/* Validates `cfg` and binds a caller-owned device workspace (256-byte aligned,
 * ws_bytes >= sr_workspace_bytes(cfg, r_max)) to a new host handle, written to
 * *out.  The workspace must stay allocated, and must not be used by anything
 * else, until sr_destroy.  A handle may be used by one stream at a time. */
sr_status sr_create(const sr_config* cfg, void* workspace, size_t ws_bytes, sr_handle** out);

/* Token selection alone (Sec. 3.2 / App. B.2).
 *  x      : [B, L, D] device; read only by SR_SEL_TOPK_L2 and SR_SEL_LAPLACIAN
 *           (the tensor the scores are taken of), may be NULL for SR_SEL_RANDOM.
 *  idx    : [B, K] int32 device output, each row strictly increasing.
 *  K_out  : host int32, receives K (may be NULL).
 * Returns SR_ERR_INVALID_ARG when keep_ratio is outside (0, 1] or K < 1.
 * The score-based selectors use the workspace for their per-token scores; the
 * random selector touches only idx. */
sr_status sr_select(sr_handle* h, const void* x, float keep_ratio, uint64_t seed,
                    int32_t* idx, int32_t* K_out, void* stream);

/* The routed encoder forward of Alg. 1.
 *  x       : [B, L, D] device input tokens.
 *  w       : HOST array of N = n1 + n2 + n3 sr_block_weights (device pointers);
 *            only read during the call.
 *  out     : [B, L, D] device output; may equal x (in place) but must not
 *            otherwise overlap it.
 *  idx_out : optional [B, K] int32 device buffer that receives the index set,
 *            or NULL.  With SR_SEL_RANDOM it is identical to sr_select's for
 *            the same arguments.  SR_SEL_TOPK_L2 ranks the output of the last
 *            dense-early block (x itself when n1 == 0); sr_select given that
 *            tensor picks the same set up to ties of the fp32 scores (the
 *            sums are added in a different order).  SR_SEL_LAPLACIAN ranks
 *            the same tensor, with the same scores as sr_select.
 * keep_ratio == 1 runs the plain dense stack (Sec. 3.4, "Architecture-agnostic design": r = 1 is the dense
 * baseline), with no selection, gather or scatter; n2 == 0 likewise routes
 * nothing.  Unselected rows of out are bit-identical to the input of the first
 * sparse block.  The delta of Eq. 9 is formed in fp32 from the last sparse
 * block's fp32 result and the stored h0, and x0 + delta is rounded once.
 * CUDA graphs: the first call of a handle (and the first call of a shape in the
 * process) sets kernel attributes and clears the handle's fault word; later
 * calls only enqueue work on `stream`, so they can be captured into a CUDA
 * graph and replayed (the keep ratio, seed and pointers are fixed in the
 * graph). */
sr_status sr_forward(sr_handle* h, const void* x, const sr_block_weights* w, float keep_ratio,
                     uint64_t seed, void* out, int32_t* idx_out, void* stream);

/* Implicit ensemble (Sec. 3, "Training and inference"; App. B): averaging the
 * outputs of forward passes with different selection seeds.  Member m is
 * exactly sr_forward(x, seeds[m]); the n1 dense-early blocks do not depend on
 * the seed, so they run once (on the handle) and their result is copied to
 * every member.  The members' selection uses the handle; their sparse-middle
 * and dense-late blocks run together as one batch of M * B samples in the
 * ensemble workspace (member m's sample b is sample m * B + b), one launch
 * sequence for all members.  When nothing is routed (keep_ratio == 1 or
 * n2 == 0) every member is the same dense forward, which runs once and is the
 * mean.
 *  seeds        : HOST array of M >= 1 selection seeds.
 *  ens_workspace: device buffer of at least sr_ensemble_workspace_bytes(cfg, M,
 *                 keep_ratio) bytes, 256-byte aligned, caller-owned (the
 *                 batch's fp32 stream and per-block buffers: the workspace of a
 *                 config with M * B samples).
 *  out          : [B, L, D] device; the mean over the members of their fp32
 *                 results, rounded once to the storage dtype.  May equal x.
 *  members_out  : optional [M, B, L, D] device; member m's output, bit-identical
 *                 to sr_forward's for seed seeds[m].  NULL to skip.
 *  idx_out      : optional [M, B, K] int32 device; member m's index set.
 * Errors as sr_forward, plus SR_ERR_INVALID_ARG for M < 1 or NULL seeds,
 * SR_ERR_UNSUPPORTED when the batch of M * B samples exceeds what the kernels
 * accept, and SR_ERR_WORKSPACE for a missing or short ensemble workspace.
 * sr_ensemble_workspace_bytes returns 0 for an invalid config or M < 1. */
size_t sr_ensemble_workspace_bytes(const sr_config* cfg, int32_t M, float max_keep_ratio);
sr_status sr_forward_ensemble(sr_handle* h, const void* x, const sr_block_weights* w,
                              float keep_ratio, const uint64_t* seeds, int32_t M,
                              void* ens_workspace, size_t ens_ws_bytes, void* out,
                              void* members_out, int32_t* idx_out, void* stream);

/* Asymmetric attention (Sec. 3.4, "Integration with generative forecasting";
 * Alg. 2): queries from one token set, keys and values from another, within
 * each sample and per head: out = softmax(q k^T / 8) v.  In the EDM model's
 * sparse stage the K routed tokens attend over the full L-token conditioning
 * sequence, O(K L D) instead of O(L^2 D).  Standalone: no handle.
 *  q     : [B, Tq, D] bf16 device, head h in columns [64h, 64h + 64).
 *  kv    : [B, Tkv, 2D] bf16 device: k in columns [0, D), v in [D, 2D).
 *  out   : [B, Tq, D] bf16 device; must not overlap q or kv.
 *  fault : optional device uint32 word; a wait of the kernel that runs out
 *          sets its bit 0 (as sr_device_fault reports for the encoder).  NULL
 *          to ignore.
 * D = 64 * heads (heads 1..32); q, kv and out 16-byte aligned.  Host-checked
 * errors: SR_ERR_INVALID_ARG (NULL or misaligned pointers, sizes below 1,
 * overlap), SR_ERR_UNSUPPORTED (heads out of range or sizes past 2^31 elements). */
sr_status sr_cross_attention(const void* q, const void* kv, int32_t B, int32_t Tq, int32_t Tkv,
                             int32_t heads, void* out, uint32_t* fault, void* stream);

/* sr_forward from and to HOST memory: copies x_host ([B, L, D], preferably
 * pinned) into the caller's device buffer `dev_xout`, runs sr_forward in place
 * on it, and copies the result back into out_host.  All three steps are
 * enqueued on `stream`; out_host is valid after the stream synchronises. */
sr_status sr_forward_host(sr_handle* h, const void* x_host, const sr_block_weights* w,
                          float keep_ratio, uint64_t seed, void* dev_xout, void* out_host,
                          int32_t* idx_out, void* stream);

/* ---- per-kernel tracing (CUDA events around every launch of a handle) ----
 * Kinds of launch the forward issues; the trace sums, per kind, the device time
 * between CUDA events recorded on the launching stream around each launch, the
 * launch count, and the launches' algorithmic work: flops (GEMM 2*M*N*K;
 * attention 4*B*heads*T^2*64 for q k^T and P v) and HBM bytes (every operand
 * read once, every result written once).  Tracing is off by default, adds two
 * event records per launch when on, and records nothing while the stream is
 * being captured into a CUDA graph. */
typedef enum {
  SR_KERN_COPY = 0,          /* stream conversions and copies: widen x to the fp32
                                stream, narrow it to out, ensemble sums */
  SR_KERN_SELECT = 1,        /* token selection (and the top-K norms when not fused into FC2) */
  SR_KERN_GATHER = 2,        /* h0 = x[:, I, :] (Eq. 8), fused with LN1 of the first
                                sparse block: reads the selected rows, writes h0 and LN1 */
  SR_KERN_LAYERNORM = 3,
  SR_KERN_GEMM_QKV = 4,      /* LN1(x) Wqkv^T + bqkv */
  SR_KERN_ATTENTION = 5,     /* softmax(q k^T / 8) v per (sample, head) */
  SR_KERN_GEMM_OUT = 6,      /* x += A Wo^T + bo */
  SR_KERN_GEMM_FC1 = 7,      /* GELU(LN2(x) W1^T + b1) */
  SR_KERN_GEMM_FC2 = 8,      /* x += U W2^T + b2 */
  SR_KERN_GEMM_FC2_SCATTER = 9,  /* last sparse block: FC2 + delta scatter (Eq. 9) */
  SR_KERN_COUNT = 10
} sr_kernel_kind;

typedef struct {
  double ms;         /* summed event-timed device milliseconds */
  int64_t launches;
  double flops;      /* algorithmic floating-point operations */
  double bytes;      /* algorithmic HBM bytes */
} sr_trace_entry;

/* Turns tracing on (1) or off (0) for later calls on this handle. */
sr_status sr_trace_enable(sr_handle* h, int enable);

/* Waits for the traced launches to finish and writes the per-kind sums since the
 * last reset into out[0 .. SR_KERN_COUNT-1] (host array).  reset != 0 clears
 * them afterwards. */
sr_status sr_trace_read(sr_handle* h, sr_trace_entry* out, int reset);

/* Releases the handle (not the workspace, which the caller owns).  NULL is a no-op. */
sr_status sr_destroy(sr_handle* h);

/* ---- allocation-free variant of the top-K L2-norm selector ---------------
 * The paper has no counterpart of this call; it exists for callers that cannot
 * allocate device memory: a plugin running inside a host framework that owns
 * the GPU's memory pool and hands it no workspace, or a latency-critical path
 * on which cudaMalloc's implicit device synchronisation is not acceptable.
 * It computes exactly what sr_select computes with SR_SEL_TOPK_L2 for the same
 * x, B, L, D, dtype and keep_ratio, but needs no handle and no workspace: its
 * per-token score scratch is a static device array of 1,048,576 floats (4 MiB)
 * compiled into this library, which every GPU that loads the library keeps
 * until the process exits.
 *  x        : [B, L, D] device, dtype storage (SR_F32 / SR_BF16), 16-byte aligned.
 *  idx      : [B, K] int32 device output, each row strictly increasing.
 *  K_out    : host int32, receives K = floor(L * keep_ratio) (may be NULL).
 * Returns SR_ERR_UNSUPPORTED when B * L exceeds 1,048,576 (or L or D exceed
 * what the selection kernels support), SR_ERR_INVALID_ARG for bad pointers,
 * dtype or ratio, before any launch.  Calls no cudaMalloc, cudaFree or other
 * allocating routine.  Every call looks up the static array's device address
 * in the current context (cudaGetSymbolAddress; the first call on a device
 * also loads the library's module there), so make the first call on each
 * device before any stream capture.  All calls share the one array and it keeps the last
 * call's scores; each call overwrites every score it reads, so nothing has to
 * start at zero, but calls whose work overlaps on the GPU (other streams, or
 * other host threads on the same device) race on it and must be serialised
 * by the caller. */
sr_status sr_select_topk_l2_static(const void* x, int32_t B, int32_t L, int32_t D, int32_t dtype,
                                   float keep_ratio, int32_t* idx, int32_t* K_out, void* stream);

/* Static description of a status code. */
const char* sr_status_string(sr_status s);

/* Reads the handle's device fault word (kept in its workspace) into *fault
 * (host) after the work enqueued on `stream` so far, resetting it when
 * clear != 0.  Bit 0 set means a tensor-core kernel of that handle gave up
 * waiting on one of its pipeline barriers (each wait is bounded to 2 s) and
 * returned early, so the outputs of that call are invalid.  The handle's first
 * sr_forward zeroes the word; afterwards it stays set until cleared here.
 * Synchronises `stream`. */
sr_status sr_device_fault(sr_handle* h, uint32_t* fault, int clear, void* stream);

/* The last CUDA or validation message recorded on this thread ("" if none). */
const char* sr_last_error_message(void);

/* ---- testing hooks -----------------------------------------------------
 * The paper has no counterpart of these calls; they exist so that the error
 * paths can be tested without making a GPU fail. */

/* Host-side fault injection.  From this call on, the CUDA call with index n
 * (0-based) among those the entry points above make through their checked
 * path (kernel launches, stream-ordered copies and memsets, stream and event
 * synchronisation) is not made and reports cudaErrorLaunchFailure instead; the
 * entry point then returns SR_ERR_CUDA with a message naming the step and
 * "[injected ...]", and enqueues nothing after it.  n < 0 turns injection off.
 * Process-wide; resets the count read by sr_debug_enqueue_count. */
void sr_debug_fail_enqueue(int64_t n);

/* Checked CUDA calls attempted (made, or failed by injection) since the last
 * sr_debug_fail_enqueue. */
int64_t sr_debug_enqueue_count(void);

/* Runs the bounded mbarrier wait of the tensor-core kernels on a barrier that
 * nothing arrives at, with a limit of limit_us microseconds (1 .. 1000000)
 * instead of the kernels' 2 s: one thread of one CTA waits, gives up, sets bit 0
 * of *fault (device) as the kernels do, and stores the nanoseconds it waited in
 * *waited_ns (device).  No TMA or tensor memory is involved; the context stays
 * usable.  Asynchronous on `stream`. */
sr_status sr_selftest_wait_timeout(uint32_t* fault, uint32_t limit_us, uint64_t* waited_ns,
                                   void* stream);

#ifdef __cplusplus
}
#endif

#endif /* SPARSE_RESLIM_H */
