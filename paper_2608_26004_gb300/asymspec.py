"""Python binding of the C ABI in include/asymspec.h.

Argument marshalling only: every function below passes plain integers
(device addresses, sizes) to ``libasymspec.so``; all of the step runs in the
library's CUDA kernels.  The functions keep the C names without the
``asymspec_`` prefix.  ``FuseVerify`` is a convenience holder for PyTorch
users: it owns a workspace tensor and extracts ``data_ptr()`` and the current
CUDA stream from tensors.  There is no fallback: if the library is missing
or fails to load, every call raises.
"""
from __future__ import annotations

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libasymspec.so")

OK = 0
ERR_INVALID_ARG = -1
ERR_UNSUPPORTED = -2
ERR_MISALIGNED = -3
ERR_WORKSPACE = -4
ERR_CUDA = -5
ERR_TOO_LARGE = -6
ERR_SCRATCH_LIMIT = -7

STATIC_MAX_ROWS = 8192  # B*(K+1) limit of fuse_verify_static
STATIC_SCRATCH_BYTES = 4 << 20  # size of fuse_verify_static's scratch array
DRAFT_MAX_V = 1 << 20  # largest V draft_sample takes

DATA_BAD_TOKEN = 0x1
DATA_NONFINITE = 0x2
DATA_BAD_PROB = 0x4
DATA_BAD_UNIFORM = 0x8
DATA_TIMEOUT = 0x10
DATA_BAD_MAP = 0x20

FP32 = 0
BF16 = 1
MODE_GREEDY = 0
MODE_STOCHASTIC = 1
DIV_JSD = 0
DIV_NONE = 1
DIV_KL = 2
DIV_LAMBDA = 3

# Every function include/asymspec.h declares.
EXPORTED = (
    "asymspec_default_gate_params",
    "asymspec_workspace_bytes",
    "asymspec_workspace_reset",
    "asymspec_fuse_verify",
    "asymspec_fuse_verify_ex",
    "asymspec_fuse_verify_static",
    "asymspec_host_scratch_bytes",
    "asymspec_fuse_verify_host",
    "asymspec_draft_sample",
    "asymspec_xvocab_gather_scratch_bytes",
    "asymspec_xvocab_workspace_bytes",
    "asymspec_xvocab_gather",
    "asymspec_fuse_verify_xvocab",
    "asymspec_plan",
    "asymspec_status_string",
    "asymspec_last_cuda_error",
    "asymspec_version",
)


class GateParams(ctypes.Structure):
    _fields_ = [("gamma", ctypes.c_float), ("beta", ctypes.c_float),
                ("lambda_", ctypes.c_float), ("mode", ctypes.c_int32),
                ("divergence", ctypes.c_int32), ("fuse_bonus", ctypes.c_int32),
                ("flags", ctypes.c_int32)]


DELTA_AB = 0   # delta = a - b (Eq. 1)
DELTA_A = 1    # delta = a (raw-augmented)
DELTA_TB = 2   # delta = t - b (SCD-style)

TEST_COPY_GIVE_UP = 1  # asymspec_launch_opts.test_flags: the copy waits give up at once

KERNEL_AUTO = 0
KERNEL_GENERIC = 1
KERNEL_TMA = 2


class LaunchOpts(ctypes.Structure):
    _fields_ = [("cluster_size", ctypes.c_int32), ("block_threads", ctypes.c_int32),
                ("kernel", ctypes.c_int32), ("test_flags", ctypes.c_int32),
                ("timing_begin", ctypes.c_void_p), ("timing_end", ctypes.c_void_p)]


class LaunchInfo(ctypes.Structure):
    _fields_ = [("cluster_size", ctypes.c_int32), ("block_threads", ctypes.c_int32),
                ("slice_elems", ctypes.c_int32), ("smem_bytes", ctypes.c_int32),
                ("ctas", ctypes.c_int64), ("vector_path", ctypes.c_int32),
                ("max_active_clusters", ctypes.c_int32), ("kernel", ctypes.c_int32),
                ("launches", ctypes.c_int32), ("row_kernel", ctypes.c_int32)]


class AsymSpecError(RuntimeError):
    def __init__(self, status: int, where: str):
        msg = status_string(status)
        if status == ERR_CUDA:
            msg += f" (cudaError {last_cuda_error()})"
        super().__init__(f"{where}: {msg} [{status}]")
        self.status = status


_lib = None
_P = ctypes.c_void_p
_I = ctypes.c_int


def lib():
    """The loaded library (raises if it is missing: build it first)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing; build it with "
                           "`python -c 'import __graft_entry__ as g; g.build()'`")
    L = ctypes.CDLL(LIB_PATH)
    L.asymspec_default_gate_params.argtypes = [ctypes.POINTER(GateParams)]
    L.asymspec_default_gate_params.restype = None
    L.asymspec_workspace_bytes.argtypes = [_I, _I, _I]
    L.asymspec_workspace_bytes.restype = ctypes.c_size_t
    L.asymspec_workspace_reset.argtypes = [_P, ctypes.c_size_t, _P]
    L.asymspec_workspace_reset.restype = _I
    L.asymspec_fuse_verify.argtypes = [_P, _P, _P, _P, _P, _P, _I, _I, _I, _I,
                                       ctypes.POINTER(GateParams), _P, _P, _P]
    L.asymspec_fuse_verify.restype = _I
    L.asymspec_fuse_verify_ex.argtypes = [_P, _P, _P, _P, _P, _P, _I, _I, _I, _I,
                                          ctypes.POINTER(GateParams), _P, _P, _P,
                                          ctypes.c_size_t, _P, _P, _P, _P,
                                          ctypes.POINTER(LaunchOpts), _P]
    L.asymspec_fuse_verify_ex.restype = _I
    L.asymspec_fuse_verify_static.argtypes = [_P, _P, _P, _P, _P, _P, _I, _I, _I, _I,
                                              ctypes.POINTER(GateParams), _P, _P, _P]
    L.asymspec_fuse_verify_static.restype = _I
    L.asymspec_host_scratch_bytes.argtypes = [_I, _I, _I, _I]
    L.asymspec_host_scratch_bytes.restype = ctypes.c_size_t
    L.asymspec_fuse_verify_host.argtypes = [_P, _P, _P, _P, _P, _P, _I, _I, _I, _I,
                                            ctypes.POINTER(GateParams), _P, _P, _P,
                                            ctypes.c_size_t, _P]
    L.asymspec_fuse_verify_host.restype = _I
    L.asymspec_draft_sample.argtypes = [_P, _I, _I, _I, _I, _P, _P, _P, _I, _P]
    L.asymspec_draft_sample.restype = _I
    L.asymspec_xvocab_gather_scratch_bytes.argtypes = [_I, _I]
    L.asymspec_xvocab_gather_scratch_bytes.restype = ctypes.c_size_t
    L.asymspec_xvocab_workspace_bytes.argtypes = [_I, _I, _I, _I, _I, _I]
    L.asymspec_xvocab_workspace_bytes.restype = ctypes.c_size_t
    L.asymspec_xvocab_gather.argtypes = [_P, _P, _I, _P, _I, _P, _P, _I, _I, _I, _P, _P, _P,
                                         _P, _P, ctypes.c_size_t, _P]
    L.asymspec_xvocab_gather.restype = _I
    L.asymspec_fuse_verify_xvocab.argtypes = [_P, _P, _I, _P, _I, _P, _P, _I, _P, _P, _P, _I,
                                              _I, _I, ctypes.POINTER(GateParams), _P, _P, _P,
                                              _P, ctypes.c_size_t, _P, _P]
    L.asymspec_fuse_verify_xvocab.restype = _I
    L.asymspec_plan.argtypes = [_I, _I, _I, _I, ctypes.POINTER(GateParams),
                                ctypes.POINTER(LaunchOpts), ctypes.POINTER(LaunchInfo)]
    L.asymspec_plan.restype = _I
    L.asymspec_status_string.argtypes = [_I]
    L.asymspec_status_string.restype = ctypes.c_char_p
    L.asymspec_last_cuda_error.argtypes = []
    L.asymspec_last_cuda_error.restype = _I
    L.asymspec_version.argtypes = []
    L.asymspec_version.restype = _I
    _lib = L
    return L


def default_gate_params() -> GateParams:
    g = GateParams()
    lib().asymspec_default_gate_params(ctypes.byref(g))
    return g


def gate_params(gamma=0.5, beta=1.0, lam=0.1, mode=MODE_GREEDY, divergence=DIV_JSD,
                fuse_bonus=False, delta_source=DELTA_AB) -> GateParams:
    """Gate parameters; delta_source goes into the flags (bits 0-1)."""
    return GateParams(gamma, beta, lam, mode, divergence, int(bool(fuse_bonus)),
                      int(delta_source))


def workspace_bytes(B: int, K: int, V: int) -> int:
    return int(lib().asymspec_workspace_bytes(B, K, V))


def workspace_reset(workspace: int, nbytes: int, stream: int = 0) -> int:
    return lib().asymspec_workspace_reset(workspace, nbytes, stream)


def fuse_verify(logits_full, logits_comp, logits_ver, draft_tokens, draft_probs, uniforms,
                B, K, V, dtype, gate, out_accept_len, out_next_token, stream=0) -> int:
    """asymspec_fuse_verify with device addresses (ints); returns the status."""
    g = ctypes.byref(gate) if gate is not None else None
    return lib().asymspec_fuse_verify(logits_full, logits_comp, logits_ver, draft_tokens,
                                      draft_probs, uniforms, B, K, V, dtype, g,
                                      out_accept_len, out_next_token, stream)


def fuse_verify_ex(logits_full, logits_comp, logits_ver, draft_tokens, draft_probs, uniforms,
                   B, K, V, dtype, gate, out_accept_len, out_next_token, workspace,
                   workspace_nbytes, out_row_stats=None, out_row_tokens=None,
                   out_fused_logprobs=None, out_error_word=None, opts=None, stream=0) -> int:
    """asymspec_fuse_verify_ex with device addresses (ints); returns the status."""
    g = ctypes.byref(gate) if gate is not None else None
    o = ctypes.byref(opts) if opts is not None else None
    return lib().asymspec_fuse_verify_ex(
        logits_full, logits_comp, logits_ver, draft_tokens, draft_probs, uniforms, B, K, V,
        dtype, g, out_accept_len, out_next_token, workspace, workspace_nbytes, out_row_stats,
        out_row_tokens, out_fused_logprobs, out_error_word, o, stream)


def fuse_verify_static(logits_full, logits_comp, logits_ver, draft_tokens, draft_probs,
                       uniforms, B, K, V, dtype, gate, out_accept_len, out_next_token,
                       stream=0) -> int:
    """asymspec_fuse_verify_static with device addresses (ints); returns the status.

    Allocates nothing (the scratch is a static array of the library); calls
    that overlap in time on one device race on it.
    """
    g = ctypes.byref(gate) if gate is not None else None
    return lib().asymspec_fuse_verify_static(logits_full, logits_comp, logits_ver,
                                             draft_tokens, draft_probs, uniforms, B, K, V,
                                             dtype, g, out_accept_len, out_next_token, stream)


HOST_CHUNKS = 8  # chunks of batch elements asymspec_fuse_verify_host pipelines


def host_scratch_bytes(B, K, V, dtype) -> int:
    return lib().asymspec_host_scratch_bytes(B, K, V, dtype)


def fuse_verify_host(h_logits_full, h_logits_comp, h_logits_ver, h_draft_tokens, h_draft_probs,
                     h_uniforms, B, K, V, dtype, gate, h_out_accept_len, h_out_next_token,
                     d_scratch, scratch_bytes, stream=0) -> int:
    """asymspec_fuse_verify_host with host addresses (ints) for the inputs and
    outputs and a device scratch address; returns the status.  The outputs
    are written once `stream` has reached the end of the call."""
    g = ctypes.byref(gate) if gate is not None else None
    return lib().asymspec_fuse_verify_host(h_logits_full, h_logits_comp, h_logits_ver,
                                           h_draft_tokens, h_draft_probs, h_uniforms, B, K, V,
                                           dtype, g, h_out_accept_len, h_out_next_token,
                                           d_scratch, scratch_bytes, stream)


def draft_sample(logits, rows, V, dtype, mode, uniforms, out_tokens, out_probs, cluster_size=0,
                 stream=0) -> int:
    """asymspec_draft_sample with device addresses (ints); returns the status."""
    return lib().asymspec_draft_sample(logits, rows, V, dtype, mode, uniforms, out_tokens,
                                       out_probs, cluster_size, stream)


def xvocab_gather_scratch_bytes(V_d, V_v) -> int:
    return int(lib().asymspec_xvocab_gather_scratch_bytes(V_d, V_v))


def xvocab_workspace_bytes(B, K, S, V_d, V_v, dtype) -> int:
    return int(lib().asymspec_xvocab_workspace_bytes(B, K, S, V_d, V_v, dtype))


def xvocab_gather(logits_full, logits_comp, V_d, logits_ver, V_v, map_d, map_v, S, rows, dtype,
                  out_full, out_comp, out_ver, out_error_word=None, scratch=None,
                  scratch_nbytes=0, stream=0) -> int:
    """asymspec_xvocab_gather with device addresses (ints); returns the status."""
    return lib().asymspec_xvocab_gather(logits_full, logits_comp, V_d, logits_ver, V_v, map_d,
                                        map_v, S, rows, dtype, out_full, out_comp, out_ver,
                                        out_error_word, scratch, scratch_nbytes, stream)


def fuse_verify_xvocab(logits_full, logits_comp, V_d, logits_ver, V_v, map_d, map_v, S,
                       draft_index, draft_probs, uniforms, B, K, dtype, gate, out_accept_len,
                       out_next_token, out_next_index, workspace, workspace_nbytes,
                       out_error_word=None, stream=0) -> int:
    """asymspec_fuse_verify_xvocab with device addresses (ints); returns the status."""
    g = ctypes.byref(gate) if gate is not None else None
    return lib().asymspec_fuse_verify_xvocab(
        logits_full, logits_comp, V_d, logits_ver, V_v, map_d, map_v, S, draft_index,
        draft_probs, uniforms, B, K, dtype, g, out_accept_len, out_next_token, out_next_index,
        workspace, workspace_nbytes, out_error_word, stream)


def plan(B, K, V, dtype, gate=None, opts=None) -> LaunchInfo:
    info = LaunchInfo()
    st = lib().asymspec_plan(B, K, V, dtype, ctypes.byref(gate) if gate is not None else None,
                             ctypes.byref(opts) if opts is not None else None,
                             ctypes.byref(info))
    if st != OK:
        raise AsymSpecError(st, "asymspec_plan")
    return info


def status_string(status: int) -> str:
    return lib().asymspec_status_string(status).decode()


def last_cuda_error() -> int:
    return int(lib().asymspec_last_cuda_error())


def version() -> int:
    return int(lib().asymspec_version())


# ----------------------------------------------------------------- PyTorch

def _ptr(t):
    return 0 if t is None else int(t.data_ptr())


class FuseVerify:
    """Holds a zeroed workspace for batches of up to B_max elements with K drafts.

    ``__call__`` takes CUDA tensors ([B, K+1, V] logits as float32 or
    bfloat16, int32 tokens, float32 probabilities and uniforms) and enqueues
    the step on the current stream.  Outputs are returned as tensors.  The
    workspace is sized for V_max vocabulary entries, or for the first call's
    V when V_max is not given (and grown, zeroed, for a larger V).
    """

    def __init__(self, B_max: int, K: int, device=None, V_max: int | None = None):
        self.B_max, self.K = B_max, K
        self.device = device
        self.V_ws = 0
        self.nbytes = 0
        self.workspace = None
        if V_max is not None:
            self._ensure(V_max)

    def _ensure(self, V: int):
        import torch
        if self.workspace is not None and V <= self.V_ws:
            return
        self.V_ws = V
        self.nbytes = workspace_bytes(self.B_max, self.K, V)
        self.workspace = torch.zeros(self.nbytes, dtype=torch.uint8,
                                     device=torch.device(self.device or "cuda"))

    def __call__(self, logits_full, logits_comp, logits_ver, draft_tokens, draft_probs=None,
                 uniforms=None, *, gamma=0.5, beta=1.0, lam=0.1, mode=MODE_GREEDY,
                 divergence=DIV_JSD, fuse_bonus=False, row_stats=False, row_tokens=False,
                 fused_logprobs=False, cluster_size=0, kernel=KERNEL_AUTO, out=None,
                 delta_source=DELTA_AB, test_flags=0, block_threads=0):
        import torch
        B, K1, V = logits_full.shape
        K = K1 - 1
        if K != self.K or B > self.B_max:
            raise ValueError("batch does not fit this workspace")
        self._ensure(V)
        if logits_full.dtype == torch.float32:
            dtype = FP32
        elif logits_full.dtype == torch.bfloat16:
            dtype = BF16
        else:
            raise TypeError("logits must be float32 or bfloat16")
        for x in (logits_full, logits_comp, logits_ver):
            if not x.is_cuda or not x.is_contiguous() or x.dtype != logits_full.dtype \
                    or tuple(x.shape) != (B, K1, V):
                raise ValueError("logits must be contiguous CUDA tensors of one shape and dtype")
        dev = logits_full.device
        res = out if out is not None else {}
        if "accept_len" not in res:
            res["accept_len"] = torch.empty(B, dtype=torch.int32, device=dev)
            res["next_token"] = torch.empty(B, dtype=torch.int32, device=dev)
            res["error_word"] = torch.zeros(1, dtype=torch.int32, device=dev)
        if row_stats and "row_stats" not in res:
            res["row_stats"] = torch.empty(B, K1, 8, dtype=torch.float32, device=dev)
        if row_tokens and "row_tokens" not in res:
            res["row_tokens"] = torch.empty(B, K1, 2, dtype=torch.int32, device=dev)
        if fused_logprobs and "fused_logprobs" not in res:
            res["fused_logprobs"] = torch.empty(B, K1, V, dtype=torch.float32, device=dev)
        gate = gate_params(gamma, beta, lam, mode, divergence, fuse_bonus, delta_source)
        opts = (LaunchOpts(cluster_size, block_threads, kernel, test_flags)
                if (cluster_size or kernel or test_flags or block_threads) else None)
        stream = torch.cuda.current_stream(dev).cuda_stream
        st = fuse_verify_ex(
            _ptr(logits_full), _ptr(logits_comp), _ptr(logits_ver), _ptr(draft_tokens),
            _ptr(draft_probs), _ptr(uniforms), B, K, V, dtype, gate,
            _ptr(res["accept_len"]), _ptr(res["next_token"]), _ptr(self.workspace),
            self.nbytes, _ptr(res.get("row_stats") if row_stats else None),
            _ptr(res.get("row_tokens") if row_tokens else None),
            _ptr(res.get("fused_logprobs") if fused_logprobs else None),
            _ptr(res["error_word"]), opts, stream)
        if st != OK:
            raise AsymSpecError(st, "asymspec_fuse_verify_ex")
        return res


def draft_tokens(logits, uniforms=None, *, mode=MODE_GREEDY, cluster_size=0, out=None):
    """The drafter's draw for CUDA tensors: logits [..., V] (float32 or
    bfloat16, contiguous), uniforms [...] float32 for sampling.  Returns
    (tokens int32, probs float32) of the leading shape, enqueued on the
    current stream; ``out`` may pass the two tensors to fill."""
    import torch
    if logits.dtype == torch.float32:
        dtype = FP32
    elif logits.dtype == torch.bfloat16:
        dtype = BF16
    else:
        raise TypeError("logits must be float32 or bfloat16")
    if not logits.is_cuda or not logits.is_contiguous():
        raise ValueError("logits must be a contiguous CUDA tensor")
    lead, V = tuple(logits.shape[:-1]), int(logits.shape[-1])
    rows = 1
    for n in lead:
        rows *= n
    if mode == MODE_STOCHASTIC:
        if uniforms is None or uniforms.dtype != torch.float32 or not uniforms.is_cuda \
                or not uniforms.is_contiguous() or uniforms.numel() != rows:
            raise ValueError("sampling takes one contiguous float32 CUDA uniform per row")
    dev = logits.device
    tokens, probs = out if out is not None else (
        torch.empty(lead, dtype=torch.int32, device=dev),
        torch.empty(lead, dtype=torch.float32, device=dev))
    stream = torch.cuda.current_stream(dev).cuda_stream
    st = draft_sample(_ptr(logits), rows, V, dtype, mode,
                      _ptr(uniforms) if mode == MODE_STOCHASTIC else 0,
                      _ptr(tokens), _ptr(probs), cluster_size, stream)
    if st != OK:
        raise AsymSpecError(st, "asymspec_draft_sample")
    return tokens, probs
