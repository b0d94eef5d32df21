"""Python binding of the libelsaa C ABI (include/elsaa.h).

Argument marshalling only: every step of the operator runs in the CUDA
kernels of libelsaa.so. PyTorch provides device memory and streams. The
functions keep the C names. If the library has not been built, every call
raises RuntimeError; there is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os

import torch

from .build import LIB

ELSAA_OK = 0
ELSAA_ERR_INVALID_ARG = 1
ELSAA_ERR_UNSUPPORTED = 2
ELSAA_ERR_WORKSPACE = 3
ELSAA_ERR_CUDA = 4
ELSAA_ERR_DEVICE = 5
ELSAA_BF16 = 0
ELSAA_FP32 = 1
ELSAA_IMPL_AUTO = 0
ELSAA_IMPL_SIMT = 1

SYMBOLS = ("elsaa_workspace_size", "elsaa_forward", "elsaa_check_status",
           "elsaa_last_error", "elsaa_abi_version", "elsaa_profile_start",
           "elsaa_profile_stop", "elsaa_forward_noalloc",
           "elsaa_backward_workspace_size", "elsaa_backward",
           "elsaa_gates_workspace_size", "elsaa_gates",
           "elsaa_selftest_wait_timeout", "elsaa_forward_race_summaries",
           "elsaa_check_status_noalloc",
           "elsaa_selftest_wait_timeout_noalloc", "elsaa_causal_levels",
           "elsaa_causal_index_lists", "elsaa_forward_selected_keys",
           "elsaa_forward_gated_workspace_size", "elsaa_forward_gated")
# Size of the fixed scratch array behind elsaa_forward_noalloc.
ELSAA_STATIC_WORKSPACE_BYTES = 64 << 20


class elsaa_params(ctypes.Structure):
    """Mirror of struct elsaa_params (field order and types must match)."""
    _fields_ = [
        ("B", ctypes.c_int), ("H", ctypes.c_int), ("N", ctypes.c_int),
        ("d_h", ctypes.c_int), ("dtype", ctypes.c_int),
        ("causal", ctypes.c_int), ("block_size", ctypes.c_int),
        ("sort_bits", ctypes.c_int), ("gray_order", ctypes.c_int),
        ("race_tables", ctypes.c_int), ("race_bits", ctypes.c_int),
        ("beta", ctypes.c_float), ("eps", ctypes.c_float),
        ("scale", ctypes.c_float), ("lam", ctypes.c_float),
        ("fusion_mode", ctypes.c_int), ("impl", ctypes.c_int),
        ("neighbor_blocks", ctypes.c_int), ("causal_chunk", ctypes.c_int),
        ("causal_base_len", ctypes.c_int), ("out_fp32", ctypes.c_int),
        ("selector", ctypes.c_int), ("topk", ctypes.c_int),
        ("topk_blocks", ctypes.c_int),
    ]


class elsaa_gate_mlp(ctypes.Structure):
    """Mirror of struct elsaa_gate_mlp (device pointers as integers)."""
    _fields_ = [
        ("hidden", ctypes.c_int), ("w1", ctypes.c_void_p),
        ("b1", ctypes.c_void_p), ("w2", ctypes.c_void_p),
        ("b2", ctypes.c_void_p), ("w_lambda", ctypes.c_void_p),
        ("b_lambda", ctypes.c_void_p), ("c_lambda", ctypes.c_void_p),
        ("lambda_min", ctypes.c_float),
    ]


class elsaa_kernel_stat(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 32), ("launches", ctypes.c_int),
                ("total_ms", ctypes.c_double)]


class ElsaaError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__("libelsaa error %d: %s" % (code, msg))
        self.code = code


_lib = None


def load_library(path: str = LIB) -> ctypes.CDLL:
    """Load libelsaa.so (built in-tree by build.build())."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(
            "libelsaa.so is not built (%s); run "
            "`python -c 'import __graft_entry__ as g; g.build()'`" % path)
    L = ctypes.CDLL(path)
    vp = ctypes.c_void_p
    L.elsaa_workspace_size.argtypes = [ctypes.POINTER(elsaa_params),
                                       ctypes.POINTER(ctypes.c_size_t)]
    L.elsaa_workspace_size.restype = ctypes.c_int
    L.elsaa_forward.argtypes = [ctypes.POINTER(elsaa_params)] + [vp] * 14 + [
        ctypes.c_size_t, vp]
    L.elsaa_forward.restype = ctypes.c_int
    L.elsaa_check_status.argtypes = [vp, vp]
    L.elsaa_check_status.restype = ctypes.c_int
    L.elsaa_last_error.argtypes = []
    L.elsaa_last_error.restype = ctypes.c_char_p
    L.elsaa_abi_version.argtypes = []
    L.elsaa_abi_version.restype = ctypes.c_int
    L.elsaa_forward_noalloc.argtypes = [ctypes.POINTER(elsaa_params)] + [
        vp] * 13 + [vp]
    L.elsaa_forward_noalloc.restype = ctypes.c_int
    L.elsaa_profile_start.argtypes = []
    L.elsaa_profile_start.restype = ctypes.c_int
    L.elsaa_profile_stop.argtypes = [ctypes.POINTER(elsaa_kernel_stat),
                                     ctypes.c_int,
                                     ctypes.POINTER(ctypes.c_int)]
    L.elsaa_profile_stop.restype = ctypes.c_int
    L.elsaa_backward_workspace_size.argtypes = [
        ctypes.POINTER(elsaa_params), ctypes.POINTER(ctypes.c_size_t)]
    L.elsaa_backward_workspace_size.restype = ctypes.c_int
    L.elsaa_backward.argtypes = [ctypes.POINTER(elsaa_params)] + [vp] * 18 + [
        ctypes.c_size_t, vp]
    L.elsaa_forward_race_summaries.argtypes = [
        ctypes.POINTER(elsaa_params), vp, ctypes.c_size_t, vp, vp, vp]
    L.elsaa_forward_race_summaries.restype = ctypes.c_int
    L.elsaa_backward.restype = ctypes.c_int
    L.elsaa_gates_workspace_size.argtypes = [
        ctypes.POINTER(elsaa_params), ctypes.POINTER(elsaa_gate_mlp),
        ctypes.POINTER(ctypes.c_size_t)]
    L.elsaa_gates_workspace_size.restype = ctypes.c_int
    L.elsaa_gates.argtypes = [ctypes.POINTER(elsaa_params),
                              ctypes.POINTER(elsaa_gate_mlp)] + [vp] * 4 + [
        ctypes.c_size_t, vp]
    L.elsaa_gates.restype = ctypes.c_int
    L.elsaa_selftest_wait_timeout.argtypes = [vp, ctypes.c_size_t,
                                              ctypes.c_int, vp]
    L.elsaa_selftest_wait_timeout.restype = ctypes.c_int
    L.elsaa_causal_levels.argtypes = [ctypes.POINTER(elsaa_params),
                                      ctypes.POINTER(ctypes.c_int)]
    L.elsaa_causal_levels.restype = ctypes.c_int
    L.elsaa_causal_index_lists.argtypes = [ctypes.POINTER(elsaa_params), vp,
                                           ctypes.c_size_t, vp, vp]
    L.elsaa_causal_index_lists.restype = ctypes.c_int
    L.elsaa_forward_gated_workspace_size.argtypes = [
        ctypes.POINTER(elsaa_params), ctypes.POINTER(elsaa_gate_mlp),
        ctypes.POINTER(ctypes.c_size_t)]
    L.elsaa_forward_gated_workspace_size.restype = ctypes.c_int
    L.elsaa_forward_gated.argtypes = [
        ctypes.POINTER(elsaa_params), ctypes.POINTER(elsaa_gate_mlp)] + [
        vp] * 14 + [ctypes.c_size_t, vp]
    L.elsaa_forward_gated.restype = ctypes.c_int
    L.elsaa_forward_selected_keys.argtypes = [
        ctypes.POINTER(elsaa_params), vp, ctypes.c_size_t, vp, vp]
    L.elsaa_forward_selected_keys.restype = ctypes.c_int
    L.elsaa_check_status_noalloc.argtypes = [vp]
    L.elsaa_check_status_noalloc.restype = ctypes.c_int
    L.elsaa_selftest_wait_timeout_noalloc.argtypes = [ctypes.c_int, vp]
    L.elsaa_selftest_wait_timeout_noalloc.restype = ctypes.c_int
    _lib = L
    return L


def elsaa_last_error() -> str:
    return load_library().elsaa_last_error().decode()


def elsaa_abi_version() -> int:
    return load_library().elsaa_abi_version()


def _check(rc: int):
    if rc != ELSAA_OK:
        raise ElsaaError(rc, elsaa_last_error())


def make_params(B, H, N, d_h, dtype="bf16", block_size=64, sort_bits=5,
                gray_order=1, race_tables=4, race_bits=4, beta=1.0, eps=1e-6,
                scale=0.0, lam=1.0, fusion_mode=0, causal=0,
                impl=ELSAA_IMPL_AUTO, neighbor_blocks=0, causal_chunk=128,
                causal_base_len=4096, out_fp32=0, selector=0, topk=0,
                topk_blocks=1) -> elsaa_params:
    dt = {"bf16": ELSAA_BF16, "fp32": ELSAA_FP32}[dtype] if isinstance(
        dtype, str) else int(dtype)
    return elsaa_params(B, H, N, d_h, dt, causal, block_size, sort_bits,
                        gray_order, race_tables, race_bits, beta, eps, scale,
                        lam, fusion_mode, impl, neighbor_blocks, causal_chunk,
                        causal_base_len, out_fp32, selector, topk,
                        topk_blocks)


def params_for(wl, **over) -> elsaa_params:
    """Parameters of a Workload (paper_2607_20214_gb300.workloads)."""
    kw = dict(B=wl.B, H=wl.H, N=wl.N, d_h=wl.d_h, dtype=wl.dtype,
              block_size=wl.block, sort_bits=wl.sort_bits,
              gray_order=wl.gray_order, race_tables=wl.race_tables,
              race_bits=wl.race_bits, beta=wl.beta, eps=wl.eps,
              lam=wl.lam, fusion_mode=wl.fusion_mode, causal=wl.causal,
              neighbor_blocks=wl.neighbor_blocks,
              causal_chunk=wl.causal_chunk,
              causal_base_len=wl.causal_base_len,
              selector=wl.selector, topk=wl.topk,
              topk_blocks=wl.topk_blocks)
    kw.update(over)
    return make_params(**kw)


def elsaa_workspace_size(params: elsaa_params) -> int:
    n = ctypes.c_size_t(0)
    _check(load_library().elsaa_workspace_size(ctypes.byref(params),
                                               ctypes.byref(n)))
    return n.value


def _ptr(t, name, dtype=None, numel=None, device=None):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        raise TypeError("%s must be a torch.Tensor" % name)
    if device is not None and t.device != device:
        raise ValueError("%s must be on %s (got %s)" % (name, device,
                                                        t.device))
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)
    if dtype is not None and t.dtype != dtype:
        raise ValueError("%s must be %s (got %s)" % (name, dtype, t.dtype))
    if numel is not None and t.numel() != numel:
        raise ValueError("%s must have %d elements (got %d)" % (
            name, numel, t.numel()))
    return t.data_ptr()


def new_workspace(params: elsaa_params, device) -> torch.Tensor:
    """Caller-owned scratch of elsaa_workspace_size bytes (256-aligned)."""
    n = elsaa_workspace_size(params)
    return torch.empty(max(n, 256), dtype=torch.uint8, device=device)


def elsaa_forward(params: elsaa_params, q, k, v, w_sort, w_race,
                  lambda_tok=None, gates=None, o=None, log_d_sparse=None,
                  d_lr=None, m_sparse=None, perm_q=None, perm_k=None,
                  workspace=None, stream=None):
    """Enqueue elsaa_forward on `stream` (default: torch's current stream).

    Tensors are device tensors laid out as in include/elsaa.h. Returns o
    (allocated here when not given). Raises ElsaaError on a non-zero return.
    """
    lib = load_library()
    dev = q.device
    if dev.type != "cuda":
        raise ValueError("q must be a CUDA tensor")
    tdt = torch.float32 if params.dtype == ELSAA_FP32 else torch.bfloat16
    odt = torch.float32 if params.out_fp32 else tdt
    BHN = params.B * params.H * params.N
    nqkv = BHN * params.d_h
    if o is None:
        o = torch.empty(q.shape, dtype=odt, device=dev)
    if workspace is None:
        workspace = new_workspace(params, dev)
    if stream is None:
        stream = torch.cuda.current_stream(dev)
    sp = stream.cuda_stream if hasattr(stream, "cuda_stream") else stream
    args = [
        _ptr(q, "q", tdt, nqkv, dev), _ptr(k, "k", tdt, nqkv, dev),
        _ptr(v, "v", tdt, nqkv, dev),
        _ptr(w_sort, "w_sort", torch.float32,
             params.H * params.sort_bits * params.d_h, dev)
        if params.sort_bits > 0 else None,
        _ptr(w_race, "w_race", torch.float32,
             params.H * params.race_tables * params.race_bits * params.d_h,
             dev),
        _ptr(lambda_tok, "lambda_tok", torch.float32, BHN, dev),
        _ptr(gates, "gates", torch.float32, 2 * BHN, dev),
        _ptr(o, "o", odt, nqkv, dev),
        _ptr(log_d_sparse, "log_d_sparse", torch.float32, BHN, dev),
        _ptr(d_lr, "d_lr", torch.float32, BHN, dev),
        _ptr(m_sparse, "m_sparse", torch.float32, BHN, dev),
        _ptr(perm_q, "perm_q", torch.int32, BHN, dev),
        _ptr(perm_k, "perm_k", torch.int32, BHN, dev),
        _ptr(workspace, "workspace", None, None, dev),
    ]
    rc = lib.elsaa_forward(ctypes.byref(params), *args,
                           workspace.numel() * workspace.element_size(), sp)
    _check(rc)
    return o


def elsaa_backward_workspace_size(params: elsaa_params) -> int:
    n = ctypes.c_size_t(0)
    _check(load_library().elsaa_backward_workspace_size(ctypes.byref(params),
                                                        ctypes.byref(n)))
    return n.value


def elsaa_forward_race_summaries(params: elsaa_params, workspace,
                                 race_A=None, race_B=None, stream=None):
    """Copy the RACE summaries A [B, H, r], B [B, H, r, d_h] (fp32) of the
    last elsaa_forward on `workspace` into race_A, race_B (allocated here
    when not given); returns (race_A, race_B)."""
    lib = load_library()
    dev = workspace.device
    r = params.race_tables << params.race_bits
    BH = params.B * params.H
    if race_A is None:
        race_A = torch.empty((params.B, params.H, r), dtype=torch.float32,
                             device=dev)
    if race_B is None:
        race_B = torch.empty((params.B, params.H, r, params.d_h),
                             dtype=torch.float32, device=dev)
    if stream is None:
        stream = torch.cuda.current_stream(dev)
    sp = stream.cuda_stream if hasattr(stream, "cuda_stream") else stream
    rc = lib.elsaa_forward_race_summaries(
        ctypes.byref(params), _ptr(workspace, "workspace", None, None, dev),
        workspace.numel() * workspace.element_size(),
        _ptr(race_A, "race_A", torch.float32, BH * r, dev),
        _ptr(race_B, "race_B", torch.float32, BH * r * params.d_h, dev), sp)
    _check(rc)
    return race_A, race_B


def elsaa_backward(params: elsaa_params, q, k, v, w_sort, w_race, d_o,
                   perm_q, perm_k, lambda_tok=None, gates=None, dq=None,
                   dk=None, dv=None, d_gates=None, d_lambda=None,
                   race_A=None, race_B=None, workspace=None, stream=None):
    """Enqueue elsaa_backward on `stream`; returns (dq, dk, dv) (fp32,
    allocated here when not given). perm_q, perm_k come from elsaa_forward
    on the same inputs; race_A, race_B (optional) from
    elsaa_forward_race_summaries."""
    lib = load_library()
    dev = q.device
    if dev.type != "cuda":
        raise ValueError("q must be a CUDA tensor")
    tdt = torch.float32 if params.dtype == ELSAA_FP32 else torch.bfloat16
    BHN = params.B * params.H * params.N
    nqkv = BHN * params.d_h
    r = params.race_tables << params.race_bits
    shape = tuple(q.shape)
    dq = torch.empty(shape, dtype=torch.float32, device=dev) if dq is None else dq
    dk = torch.empty(shape, dtype=torch.float32, device=dev) if dk is None else dk
    dv = torch.empty(shape, dtype=torch.float32, device=dev) if dv is None else dv
    if workspace is None:
        n = elsaa_backward_workspace_size(params)
        workspace = torch.empty(max(n, 256), dtype=torch.uint8, device=dev)
    if stream is None:
        stream = torch.cuda.current_stream(dev)
    sp = stream.cuda_stream if hasattr(stream, "cuda_stream") else stream
    args = [
        _ptr(q, "q", tdt, nqkv, dev), _ptr(k, "k", tdt, nqkv, dev),
        _ptr(v, "v", tdt, nqkv, dev),
        _ptr(w_sort, "w_sort", torch.float32, None, dev)
        if w_sort is not None else None,
        _ptr(w_race, "w_race", torch.float32,
             params.H * params.race_tables * params.race_bits * params.d_h,
             dev),
        _ptr(lambda_tok, "lambda_tok", torch.float32, BHN, dev),
        _ptr(gates, "gates", torch.float32, 2 * BHN, dev),
        _ptr(d_o, "d_o", tdt, nqkv, dev),
        _ptr(perm_q, "perm_q", torch.int32, BHN, dev),
        _ptr(perm_k, "perm_k", torch.int32, BHN, dev),
        _ptr(dq, "dq", torch.float32, nqkv, dev),
        _ptr(dk, "dk", torch.float32, nqkv, dev),
        _ptr(dv, "dv", torch.float32, nqkv, dev),
        _ptr(d_gates, "d_gates", torch.float32, 2 * BHN, dev),
        _ptr(d_lambda, "d_lambda", torch.float32, BHN, dev),
        _ptr(race_A, "race_A", torch.float32, params.B * params.H * r, dev),
        _ptr(race_B, "race_B", torch.float32,
             params.B * params.H * r * params.d_h, dev),
        _ptr(workspace, "workspace", None, None, dev),
    ]
    rc = lib.elsaa_backward(ctypes.byref(params), *args,
                            workspace.numel() * workspace.element_size(), sp)
    _check(rc)
    return dq, dk, dv


def _gate_struct(params: elsaa_params, mlp: dict, dev) -> elsaa_gate_mlp:
    H, d, g = params.H, params.d_h, int(mlp["hidden"])
    has_l = mlp.get("w_lambda") is not None
    f32 = torch.float32
    return elsaa_gate_mlp(
        g, _ptr(mlp["w1"], "w1", f32, H * g * d, dev),
        _ptr(mlp["b1"], "b1", f32, H * g, dev),
        _ptr(mlp["w2"], "w2", f32, H * 2 * g, dev),
        _ptr(mlp["b2"], "b2", f32, H * 2, dev),
        _ptr(mlp["w_lambda"], "w_lambda", f32, H * d, dev) if has_l else None,
        _ptr(mlp["b_lambda"], "b_lambda", f32, H, dev) if has_l else None,
        _ptr(mlp["c_lambda"], "c_lambda", f32, H, dev) if has_l else None,
        float(mlp.get("lambda_min", 1e-6)))


def elsaa_gates_workspace_size(params: elsaa_params, mlp: dict,
                               device=None) -> int:
    dev = mlp["w1"].device if device is None else device
    m = _gate_struct(params, mlp, dev)
    n = ctypes.c_size_t(0)
    _check(load_library().elsaa_gates_workspace_size(
        ctypes.byref(params), ctypes.byref(m), ctypes.byref(n)))
    return n.value


def elsaa_gates(params: elsaa_params, mlp: dict, q, gates=None,
                lambda_tok=None, workspace=None, stream=None):
    """Enqueue elsaa_gates on `stream`: per-token (g_sparse, g_lr) and,
    when mlp["w_lambda"] is given, lambda_i. `mlp` holds device tensors
    w1, b1, w2, b2 (and w_lambda, b_lambda, c_lambda, lambda_min) as in
    include/elsaa.h. Returns (gates [B, H, N, 2], lambda_tok [B, H, N] or
    None), allocated here when not given."""
    lib = load_library()
    dev = q.device
    if dev.type != "cuda":
        raise ValueError("q must be a CUDA tensor")
    tdt = torch.float32 if params.dtype == ELSAA_FP32 else torch.bfloat16
    BHN = params.B * params.H * params.N
    shape = (params.B, params.H, params.N)
    m = _gate_struct(params, mlp, dev)
    if gates is None:
        gates = torch.empty(shape + (2,), dtype=torch.float32, device=dev)
    if lambda_tok is None and mlp.get("w_lambda") is not None:
        lambda_tok = torch.empty(shape, dtype=torch.float32, device=dev)
    if workspace is None:
        n = elsaa_gates_workspace_size(params, mlp, dev)
        workspace = torch.empty(max(n, 256), dtype=torch.uint8, device=dev)
    if stream is None:
        stream = torch.cuda.current_stream(dev)
    sp = stream.cuda_stream if hasattr(stream, "cuda_stream") else stream
    rc = lib.elsaa_gates(
        ctypes.byref(params), ctypes.byref(m),
        _ptr(q, "q", tdt, BHN * params.d_h, dev),
        _ptr(gates, "gates", torch.float32, 2 * BHN, dev),
        _ptr(lambda_tok, "lambda_tok", torch.float32, BHN, dev),
        _ptr(workspace, "workspace", None, None, dev),
        workspace.numel() * workspace.element_size(), sp)
    _check(rc)
    return gates, lambda_tok


def elsaa_selftest_wait_timeout(workspace: torch.Tensor, limit_ms=100,
                                stream=None):
    """Enqueue the bounded-wait self-test: one wait that nothing satisfies
    runs out after limit_ms and records a timeout in the status word."""
    lib = load_library()
    if stream is None:
        stream = torch.cuda.current_stream(workspace.device)
    sp = stream.cuda_stream if hasattr(stream, "cuda_stream") else stream
    _check(lib.elsaa_selftest_wait_timeout(
        workspace.data_ptr(), workspace.numel() * workspace.element_size(),
        int(limit_ms), sp))


def elsaa_check_status(workspace: torch.Tensor, stream=None):
    """Synchronise and raise ElsaaError if a kernel recorded a fault."""
    lib = load_library()
    if stream is None:
        stream = torch.cuda.current_stream(workspace.device)
    sp = stream.cuda_stream if hasattr(stream, "cuda_stream") else stream
    _check(lib.elsaa_check_status(workspace.data_ptr(), sp))


def elsaa_profile_start():
    _check(load_library().elsaa_profile_start())


def elsaa_profile_stop() -> dict:
    """{kernel name: (launches, summed device ms)} since profile_start."""
    arr = (elsaa_kernel_stat * 64)()
    n = ctypes.c_int(0)
    _check(load_library().elsaa_profile_stop(arr, 64, ctypes.byref(n)))
    return {arr[i].name.decode(): (arr[i].launches, arr[i].total_ms)
            for i in range(n.value)}


def elsaa_forward_noalloc(params: elsaa_params, q, k, v, w_sort, w_race,
                          lambda_tok=None, gates=None, o=None,
                          log_d_sparse=None, d_lr=None, m_sparse=None,
                          perm_q=None, perm_k=None, stream=None):
    """elsaa_forward without a workspace, for callers that cannot allocate
    device memory (a host application that owns every buffer, or a path
    that must not risk the device-wide synchronisation of cudaMalloc).

    Scratch comes from the library's fixed ELSAA_STATIC_WORKSPACE_BYTES
    array, shared by all calls: order overlapping calls on one stream. The
    first call on a device may load the library's module there and should
    precede any stream capture. `o` must be given (nothing is allocated here
    either). elsaa_check_status_noalloc reads the call's status word.
    """
    lib = load_library()
    if o is None:
        raise ValueError("o must be given: elsaa_forward_noalloc allocates "
                         "nothing")
    dev = q.device
    tdt = torch.float32 if params.dtype == ELSAA_FP32 else torch.bfloat16
    odt = torch.float32 if params.out_fp32 else tdt
    BHN = params.B * params.H * params.N
    nqkv = BHN * params.d_h
    if stream is None:
        stream = torch.cuda.current_stream(dev)
    sp = stream.cuda_stream if hasattr(stream, "cuda_stream") else stream
    args = [
        _ptr(q, "q", tdt, nqkv, dev), _ptr(k, "k", tdt, nqkv, dev),
        _ptr(v, "v", tdt, nqkv, dev),
        _ptr(w_sort, "w_sort", torch.float32,
             params.H * params.sort_bits * params.d_h, dev)
        if params.sort_bits > 0 else None,
        _ptr(w_race, "w_race", torch.float32,
             params.H * params.race_tables * params.race_bits * params.d_h,
             dev),
        _ptr(lambda_tok, "lambda_tok", torch.float32, BHN, dev),
        _ptr(gates, "gates", torch.float32, 2 * BHN, dev),
        _ptr(o, "o", odt, nqkv, dev),
        _ptr(log_d_sparse, "log_d_sparse", torch.float32, BHN, dev),
        _ptr(d_lr, "d_lr", torch.float32, BHN, dev),
        _ptr(m_sparse, "m_sparse", torch.float32, BHN, dev),
        _ptr(perm_q, "perm_q", torch.int32, BHN, dev),
        _ptr(perm_k, "perm_k", torch.int32, BHN, dev),
    ]
    _check(lib.elsaa_forward_noalloc(ctypes.byref(params), *args, sp))
    return o


def _stream_ptr(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else stream


def elsaa_check_status_noalloc(stream=None):
    """elsaa_check_status for elsaa_forward_noalloc: synchronise and raise
    ElsaaError if a kernel recorded a fault in the static array's status
    word."""
    _check(load_library().elsaa_check_status_noalloc(_stream_ptr(stream)))


def elsaa_selftest_wait_timeout_noalloc(limit_ms=100, stream=None):
    """The bounded-wait self-test on the static array's status word."""
    _check(load_library().elsaa_selftest_wait_timeout_noalloc(
        int(limit_ms), _stream_ptr(stream)))


def elsaa_causal_levels(params: elsaa_params) -> int:
    """Halving levels Lv of the causal sparse branch for params."""
    n = ctypes.c_int(0)
    _check(load_library().elsaa_causal_levels(ctypes.byref(params),
                                              ctypes.byref(n)))
    return n.value


def elsaa_causal_index_lists(params: elsaa_params, workspace, lists=None,
                             stream=None):
    """Sorted orders of every SortLSH call of the last causal forward on
    `workspace`: int32 [Lv, 2, B, H, N / 2] (allocated here when not
    given; None when Lv = 0). See include/elsaa.h for the layout."""
    lv = elsaa_causal_levels(params)
    if lv == 0:
        return None
    dev = workspace.device
    shape = (lv, 2, params.B, params.H, params.N // 2)
    if lists is None:
        lists = torch.empty(shape, dtype=torch.int32, device=dev)
    n = lv * params.B * params.H * params.N
    _check(load_library().elsaa_causal_index_lists(
        ctypes.byref(params), _ptr(workspace, "workspace", None, None, dev),
        workspace.numel() * workspace.element_size(),
        _ptr(lists, "lists", torch.int32, n, dev), _stream_ptr(stream)))
    return lists


def elsaa_forward_selected_keys(params: elsaa_params, workspace, keys=None,
                                stream=None):
    """The key sets of the last top-k forward (selector = 1) on `workspace`:
    int32 [B, H, N, topk], each row's original key indices increasing
    (allocated here when not given)."""
    dev = workspace.device
    shape = (params.B, params.H, params.N, params.topk)
    if keys is None:
        keys = torch.empty(shape, dtype=torch.int32, device=dev)
    n = params.B * params.H * params.N * params.topk
    _check(load_library().elsaa_forward_selected_keys(
        ctypes.byref(params), _ptr(workspace, "workspace", None, None, dev),
        workspace.numel() * workspace.element_size(),
        _ptr(keys, "keys", torch.int32, n, dev), _stream_ptr(stream)))
    return keys


def elsaa_forward_gated_workspace_size(params: elsaa_params, mlp: dict,
                                       device=None) -> int:
    dev = mlp["w1"].device if device is None else device
    m = _gate_struct(params, mlp, dev)
    n = ctypes.c_size_t(0)
    _check(load_library().elsaa_forward_gated_workspace_size(
        ctypes.byref(params), ctypes.byref(m), ctypes.byref(n)))
    return n.value


def elsaa_forward_gated(params: elsaa_params, mlp: dict, q, k, v, w_sort,
                        w_race, o=None, log_d_sparse=None, d_lr=None,
                        m_sparse=None, perm_q=None, perm_k=None,
                        gates_out=None, lambda_out=None, workspace=None,
                        stream=None):
    """Enqueue elsaa_forward_gated: the forward with the gates and lambda
    of the gate MLP `mlp` (as for elsaa_gates) computed in the same call.
    Returns o (allocated here when not given)."""
    lib = load_library()
    dev = q.device
    tdt = torch.float32 if params.dtype == ELSAA_FP32 else torch.bfloat16
    odt = torch.float32 if params.out_fp32 else tdt
    BHN = params.B * params.H * params.N
    nqkv = BHN * params.d_h
    m = _gate_struct(params, mlp, dev)
    if o is None:
        o = torch.empty(q.shape, dtype=odt, device=dev)
    if workspace is None:
        n = elsaa_forward_gated_workspace_size(params, mlp, dev)
        workspace = torch.empty(max(n, 256), dtype=torch.uint8, device=dev)
    args = [
        _ptr(q, "q", tdt, nqkv, dev), _ptr(k, "k", tdt, nqkv, dev),
        _ptr(v, "v", tdt, nqkv, dev),
        _ptr(w_sort, "w_sort", torch.float32,
             params.H * params.sort_bits * params.d_h, dev)
        if params.sort_bits > 0 else None,
        _ptr(w_race, "w_race", torch.float32,
             params.H * params.race_tables * params.race_bits * params.d_h,
             dev),
        _ptr(o, "o", odt, nqkv, dev),
        _ptr(log_d_sparse, "log_d_sparse", torch.float32, BHN, dev),
        _ptr(d_lr, "d_lr", torch.float32, BHN, dev),
        _ptr(m_sparse, "m_sparse", torch.float32, BHN, dev),
        _ptr(perm_q, "perm_q", torch.int32, BHN, dev),
        _ptr(perm_k, "perm_k", torch.int32, BHN, dev),
        _ptr(gates_out, "gates_out", torch.float32, 2 * BHN, dev),
        _ptr(lambda_out, "lambda_out", torch.float32, BHN, dev),
        _ptr(workspace, "workspace", None, None, dev),
    ]
    _check(lib.elsaa_forward_gated(
        ctypes.byref(params), ctypes.byref(m), *args,
        workspace.numel() * workspace.element_size(), _stream_ptr(stream)))
    return o
