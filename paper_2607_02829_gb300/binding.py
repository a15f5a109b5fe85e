"""ctypes binding of the C ABI declared in include/sparse_reslim.h.

Argument marshalling only: the functions keep the C names and forward plain
pointers and sizes.  PyTorch supplies device memory and streams through the
helpers at the bottom.  Loading fails loudly when the library has not been
built; there is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libsparse_reslim.so")

SR_OK, SR_ERR_INVALID_ARG, SR_ERR_UNSUPPORTED, SR_ERR_WORKSPACE, SR_ERR_CUDA, SR_ERR_INTERNAL = range(6)
SR_F32, SR_BF16 = 0, 1
SR_SEL_RANDOM, SR_SEL_TOPK_L2, SR_SEL_LAPLACIAN = 0, 1, 2

KERNEL_KINDS = ("copy", "select", "gather", "layernorm", "gemm_qkv", "attention", "gemm_out",
                "gemm_fc1", "gemm_fc2", "gemm_fc2_scatter")


class sr_config(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("L", ctypes.c_int32), ("D", ctypes.c_int32),
                ("heads", ctypes.c_int32), ("mlp_hidden", ctypes.c_int32),
                ("n1", ctypes.c_int32), ("n2", ctypes.c_int32), ("n3", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("selector", ctypes.c_int32),
                ("shared_indices", ctypes.c_int32), ("ln_eps", ctypes.c_float),
                ("grid_w", ctypes.c_int32)]


WEIGHT_FIELDS = ("ln1_g", "ln1_b", "wqkv", "bqkv", "wo", "bo",
                 "ln2_g", "ln2_b", "w1", "b1", "w2", "b2")


class sr_block_weights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in WEIGHT_FIELDS]


class sr_trace_entry(ctypes.Structure):
    _fields_ = [("ms", ctypes.c_double), ("launches", ctypes.c_int64),
                ("flops", ctypes.c_double), ("bytes", ctypes.c_double)]


class SRError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(msg)
        self.status = status


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded CUDA library (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32, sz, st = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t, ctypes.c_int
        L.sr_keep_count.argtypes = [i32, ctypes.c_float]; L.sr_keep_count.restype = i32
        L.sr_workspace_bytes.argtypes = [ctypes.POINTER(sr_config), ctypes.c_float]
        L.sr_workspace_bytes.restype = sz
        L.sr_create.argtypes = [ctypes.POINTER(sr_config), vp, sz, ctypes.POINTER(vp)]
        L.sr_create.restype = st
        L.sr_select.argtypes = [vp, vp, ctypes.c_float, ctypes.c_uint64, vp,
                                ctypes.POINTER(i32), vp]
        L.sr_select.restype = st
        L.sr_forward.argtypes = [vp, vp, ctypes.POINTER(sr_block_weights), ctypes.c_float,
                                 ctypes.c_uint64, vp, vp, vp]
        L.sr_forward.restype = st
        L.sr_forward_host.argtypes = [vp, vp, ctypes.POINTER(sr_block_weights), ctypes.c_float,
                                      ctypes.c_uint64, vp, vp, vp, vp]
        L.sr_forward_host.restype = st
        L.sr_ensemble_workspace_bytes.argtypes = [ctypes.POINTER(sr_config), i32, ctypes.c_float]
        L.sr_ensemble_workspace_bytes.restype = sz
        L.sr_forward_ensemble.argtypes = [vp, vp, ctypes.POINTER(sr_block_weights), ctypes.c_float,
                                          ctypes.POINTER(ctypes.c_uint64), i32, vp, sz, vp, vp, vp,
                                          vp]
        L.sr_forward_ensemble.restype = st
        L.sr_cross_attention.argtypes = [vp, vp, i32, i32, i32, i32, vp, vp, vp]
        L.sr_cross_attention.restype = st
        L.sr_destroy.argtypes = [vp]; L.sr_destroy.restype = st
        L.sr_trace_enable.argtypes = [vp, ctypes.c_int]; L.sr_trace_enable.restype = st
        L.sr_trace_read.argtypes = [vp, ctypes.POINTER(sr_trace_entry), ctypes.c_int]
        L.sr_trace_read.restype = st
        L.sr_device_fault.argtypes = [vp, ctypes.POINTER(ctypes.c_uint32), ctypes.c_int, vp]
        L.sr_device_fault.restype = st
        L.sr_select_topk_l2_static.argtypes = [vp, i32, i32, i32, i32, ctypes.c_float, vp,
                                               ctypes.POINTER(i32), vp]
        L.sr_select_topk_l2_static.restype = st
        L.sr_debug_fail_enqueue.argtypes = [ctypes.c_int64]; L.sr_debug_fail_enqueue.restype = None
        L.sr_debug_enqueue_count.argtypes = []; L.sr_debug_enqueue_count.restype = ctypes.c_int64
        L.sr_selftest_wait_timeout.argtypes = [vp, ctypes.c_uint32, vp, vp]
        L.sr_selftest_wait_timeout.restype = st
        L.sr_status_string.argtypes = [st]; L.sr_status_string.restype = ctypes.c_char_p
        L.sr_last_error_message.argtypes = []; L.sr_last_error_message.restype = ctypes.c_char_p
        _lib = L
    return _lib


def _check(status: int, what: str) -> None:
    if status != SR_OK:
        L = lib()
        raise SRError(status, f"{what}: {L.sr_status_string(status).decode()} -- "
                              f"{L.sr_last_error_message().decode()}")


# ------------------------------------------------------------- raw C names
def sr_keep_count(L: int, keep_ratio: float) -> int:
    return lib().sr_keep_count(L, keep_ratio)


def sr_workspace_bytes(cfg: sr_config, max_keep_ratio: float) -> int:
    return lib().sr_workspace_bytes(ctypes.byref(cfg), max_keep_ratio)


def sr_create(cfg: sr_config, workspace: int, ws_bytes: int) -> int:
    h = ctypes.c_void_p()
    _check(lib().sr_create(ctypes.byref(cfg), workspace, ws_bytes, ctypes.byref(h)), "sr_create")
    return h.value


def sr_select(handle: int, x: int, keep_ratio: float, seed: int, idx: int, stream: int) -> int:
    K = ctypes.c_int32(0)
    _check(lib().sr_select(handle, x, keep_ratio, seed % (1 << 64), idx, ctypes.byref(K), stream),
           "sr_select")
    return K.value


def sr_forward(handle: int, x: int, weights: ctypes.Array, keep_ratio: float, seed: int,
               out: int, idx_out: Optional[int], stream: int) -> None:
    _check(lib().sr_forward(handle, x, weights, keep_ratio, seed % (1 << 64), out, idx_out, stream),
           "sr_forward")


def sr_forward_host(handle: int, x_host: int, weights: ctypes.Array, keep_ratio: float,
                    seed: int, dev_xout: int, out_host: int, idx_out: Optional[int],
                    stream: int) -> None:
    _check(lib().sr_forward_host(handle, x_host, weights, keep_ratio, seed % (1 << 64), dev_xout,
                                 out_host, idx_out, stream), "sr_forward_host")


def sr_ensemble_workspace_bytes(cfg: sr_config, M: int, max_keep_ratio: float) -> int:
    return int(lib().sr_ensemble_workspace_bytes(ctypes.byref(cfg), M, max_keep_ratio))


def sr_forward_ensemble(handle: int, x: int, weights: ctypes.Array, keep_ratio: float,
                        seeds: Sequence[int], ens_ws: int, ens_ws_bytes: int, out: int,
                        members_out: Optional[int], idx_out: Optional[int], stream: int) -> None:
    arr = (ctypes.c_uint64 * max(len(seeds), 1))(*[int(v) % (1 << 64) for v in seeds])
    _check(lib().sr_forward_ensemble(handle, x, weights, keep_ratio, arr, len(seeds), ens_ws,
                                     ens_ws_bytes, out, members_out, idx_out, stream),
           "sr_forward_ensemble")


def sr_cross_attention(q: int, kv: int, B: int, Tq: int, Tkv: int, heads: int, out: int,
                       fault: Optional[int], stream: int) -> None:
    _check(lib().sr_cross_attention(q, kv, B, Tq, Tkv, heads, out, fault, stream),
           "sr_cross_attention")


def sr_destroy(handle: Optional[int]) -> None:
    if handle:
        _check(lib().sr_destroy(handle), "sr_destroy")


def sr_trace_enable(handle: int, enable: bool) -> None:
    _check(lib().sr_trace_enable(handle, int(bool(enable))), "sr_trace_enable")


def sr_trace_read(handle: int, reset: bool = True) -> dict:
    arr = (sr_trace_entry * len(KERNEL_KINDS))()
    _check(lib().sr_trace_read(handle, arr, int(bool(reset))), "sr_trace_read")
    return {k: {"ms": e.ms, "launches": e.launches, "flops": e.flops, "bytes": e.bytes}
            for k, e in zip(KERNEL_KINDS, arr)}


def sr_device_fault(handle: int, clear: bool, stream: int) -> int:
    f = ctypes.c_uint32(0)
    _check(lib().sr_device_fault(handle, ctypes.byref(f), int(bool(clear)), stream),
           "sr_device_fault")
    return f.value


def sr_select_topk_l2_static(x: int, B: int, L: int, D: int, dtype: int, keep_ratio: float,
                             idx: int, stream: int) -> int:
    K = ctypes.c_int32(0)
    _check(lib().sr_select_topk_l2_static(x, B, L, D, dtype, keep_ratio, idx, ctypes.byref(K),
                                          stream), "sr_select_topk_l2_static")
    return K.value


def sr_debug_fail_enqueue(n: int) -> None:
    lib().sr_debug_fail_enqueue(int(n))


def sr_debug_enqueue_count() -> int:
    return int(lib().sr_debug_enqueue_count())


def sr_selftest_wait_timeout(fault: int, limit_us: int, waited_ns: int, stream: int) -> None:
    _check(lib().sr_selftest_wait_timeout(fault, limit_us, waited_ns, stream),
           "sr_selftest_wait_timeout")


# ----------------------------------------------------- torch-side helpers
def make_config(B, L, D, heads, n1, n2, n3, dtype="bf16", selector="random", shared=False,
                mlp_hidden=None, ln_eps=1e-5, grid_w=0) -> sr_config:
    return sr_config(B=B, L=L, D=D, heads=heads, mlp_hidden=mlp_hidden or 4 * D, n1=n1, n2=n2,
                     n3=n3, dtype={"f32": SR_F32, "bf16": SR_BF16}[dtype],
                     selector={"random": SR_SEL_RANDOM, "topk_l2": SR_SEL_TOPK_L2,
                               "laplacian": SR_SEL_LAPLACIAN}[selector],
                     shared_indices=int(bool(shared)), ln_eps=ln_eps, grid_w=grid_w)


def weights_array(blocks: Sequence[dict]) -> ctypes.Array:
    """Host array of sr_block_weights from dicts of device tensors (kept alive by caller)."""
    arr = (sr_block_weights * len(blocks))()
    for i, blk in enumerate(blocks):
        for n in WEIGHT_FIELDS:
            t = blk[n]
            assert t.is_cuda and t.is_contiguous()
            setattr(arr[i], n, t.data_ptr())
    return arr


class Encoder:
    """Owns a handle and its workspace (a torch uint8 CUDA tensor)."""

    def __init__(self, cfg: sr_config, max_keep_ratio: float = 1.0, device="cuda"):
        import torch
        self.cfg = cfg
        nbytes = sr_workspace_bytes(cfg, max_keep_ratio)
        if nbytes == 0:
            raise SRError(SR_ERR_INVALID_ARG, "invalid config: " + lib().sr_last_error_message().decode())
        self.workspace = torch.empty(nbytes + 256, dtype=torch.uint8, device=device)
        base = self.workspace.data_ptr()
        self.ws_ptr = (base + 255) // 256 * 256
        self.ws_bytes = nbytes
        self.handle = sr_create(cfg, self.ws_ptr, nbytes)

    def close(self):
        if self.handle:
            sr_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def select(self, x, keep_ratio, seed, stream=None):
        import torch
        K = sr_keep_count(self.cfg.L, keep_ratio)
        idx = torch.empty((self.cfg.B, max(K, 1)), dtype=torch.int32, device="cuda")
        s = stream if stream is not None else torch.cuda.current_stream()
        sr_select(self.handle, x.data_ptr() if x is not None else None, keep_ratio, seed,
                  idx.data_ptr(), s.cuda_stream)
        return idx

    def forward(self, x, weights: ctypes.Array, keep_ratio, seed, out=None, want_idx=False,
                stream=None):
        import torch
        if out is None:
            out = torch.empty_like(x)
        idx = None
        if want_idx:
            K = sr_keep_count(self.cfg.L, keep_ratio)
            idx = torch.empty((self.cfg.B, max(K, 1)), dtype=torch.int32, device="cuda")
        s = stream if stream is not None else torch.cuda.current_stream()
        sr_forward(self.handle, x.data_ptr(), weights, keep_ratio, seed, out.data_ptr(),
                   idx.data_ptr() if idx is not None else None, s.cuda_stream)
        return out, idx

    def forward_ensemble(self, x, weights: ctypes.Array, keep_ratio, seeds, out=None,
                         want_members=False, want_idx=False, stream=None):
        """Mean over len(seeds) members (see sr_forward_ensemble); returns
        (out, members [M, B, L, D] or None, idx [M, B, K] or None)."""
        import torch
        M = len(seeds)
        nbytes = sr_ensemble_workspace_bytes(self.cfg, M, keep_ratio)
        if nbytes == 0:
            raise SRError(SR_ERR_INVALID_ARG, "invalid ensemble: " + lib().sr_last_error_message().decode())
        if getattr(self, "ens_ws", None) is None or self.ens_ws.numel() < nbytes + 256:
            self.ens_ws = torch.empty(nbytes + 256, dtype=torch.uint8, device="cuda")
        ptr = (self.ens_ws.data_ptr() + 255) // 256 * 256
        if out is None:
            out = torch.empty_like(x)
        members = torch.empty((M,) + tuple(x.shape), dtype=x.dtype, device="cuda") if want_members else None
        idx = None
        if want_idx:
            K = sr_keep_count(self.cfg.L, keep_ratio)
            idx = torch.empty((M, self.cfg.B, max(K, 1)), dtype=torch.int32, device="cuda")
        s = stream if stream is not None else torch.cuda.current_stream()
        sr_forward_ensemble(self.handle, x.data_ptr(), weights, keep_ratio, seeds, ptr, nbytes,
                            out.data_ptr(), members.data_ptr() if members is not None else None,
                            idx.data_ptr() if idx is not None else None, s.cuda_stream)
        return out, members, idx
