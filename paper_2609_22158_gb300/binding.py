"""ctypes binding of libstepkv.so (C ABI in include/stepkv.h).

Argument marshalling only: shapes and dtypes are checked, torch tensors are turned into device
pointers, and every step of the pass runs in the library's CUDA kernels.  PyTorch provides device
memory and streams.  There is no fallback: if the library is missing or a call fails, an exception
is raised.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass, field
from typing import List, Optional, Sequence

_PKG_DIR = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG_DIR, "libstepkv.so")

STEPKV_OK, STEPKV_EINVAL, STEPKV_ECUDA, STEPKV_ENOSPACE, STEPKV_EUNSUPPORTED, STEPKV_EDATA, STEPKV_ETIMEOUT = range(7)
NORM_MAX, NORM_NONE = 0, 1
POOL_MAX, POOL_AVG = 0, 1
BUDGET_RATIO, BUDGET_COUNT = 0, 1


class StepKVError(RuntimeError):
    def __init__(self, code: int, where: str, detail: str = ""):
        self.code = code
        super().__init__(f"{where}: status {code} ({status_string(code)}){' ' + detail if detail else ''}")


# ----------------------------------------------------------------------------- C structs
class CParams(ctypes.Structure):
    _fields_ = [("lambda_", ctypes.c_float), ("w_r", ctypes.c_float), ("w_c", ctypes.c_float),
                ("r_min", ctypes.c_float), ("r_max", ctypes.c_float), ("s_max", ctypes.c_float),
                ("eta", ctypes.c_float), ("alpha", ctypes.c_float), ("beta", ctypes.c_float),
                ("sal_norm", ctypes.c_int32), ("sal_pool", ctypes.c_int32), ("sal_pool_mode", ctypes.c_int32)]


class CBudget(ctypes.Structure):
    _fields_ = [("mode", ctypes.c_int32), ("ratio_num", ctypes.c_int32), ("ratio_den", ctypes.c_int32),
                ("count", ctypes.c_int32)]


class CSteps(ctypes.Structure):
    _fields_ = [("n_steps", ctypes.c_int32), ("valid", ctypes.c_void_p), ("gain", ctypes.c_void_p),
                ("red", ctypes.c_void_p), ("obs_sim", ctypes.c_void_p), ("reuse_in", ctypes.c_void_p),
                ("reuse_out", ctypes.c_void_p)]


class CSelOut(ctypes.Structure):
    _fields_ = [("kept_idx", ctypes.c_void_p), ("kept_cap", ctypes.c_int32), ("n_kept", ctypes.c_void_p),
                ("n_budget", ctypes.c_void_p), ("priority", ctypes.c_void_p), ("token_sal", ctypes.c_void_p),
                ("step_util", ctypes.c_void_p), ("step_count", ctypes.c_void_p), ("step_sal_sum", ctypes.c_void_p),
                ("step_sal_max", ctypes.c_void_p), ("step_kept", ctypes.c_void_p)]


class CProblem(ctypes.Structure):
    _fields_ = [("L", ctypes.c_int32), ("Hkv", ctypes.c_int32), ("Hq", ctypes.c_int32), ("d", ctypes.c_int32),
                ("T", ctypes.c_int32), ("W", ctypes.c_int32), ("n_sal_layers", ctypes.c_int32),
                ("K", ctypes.c_void_p), ("V", ctypes.c_void_p), ("kv_head_stride", ctypes.c_int64),
                ("Q", ctypes.c_void_p), ("q_head_stride", ctypes.c_int64),
                ("step_id", ctypes.c_void_p), ("prot", ctypes.c_void_p), ("pos_in", ctypes.c_void_p),
                ("steps", CSteps), ("budget", CBudget),
                ("K_out", ctypes.c_void_p), ("V_out", ctypes.c_void_p), ("out_head_stride", ctypes.c_int64),
                ("step_id_out", ctypes.c_void_p), ("pos_out", ctypes.c_void_p), ("sel", CSelOut),
                ("kv_location", ctypes.c_int32), ("out_location", ctypes.c_int32), ("K_sal", ctypes.c_void_p),
                ("sal_lse", ctypes.c_void_p)]


STEPKV_MEM_DEVICE = 0
STEPKV_MEM_HOST = 1


_lib = None

# (name, restype, argtypes) for every function declared in include/stepkv.h
_VP, _I32, _I64, _SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
SIGNATURES = {
    "stepkv_default_params": (None, [ctypes.POINTER(CParams)]),
    "stepkv_status_string": (ctypes.c_char_p, [_I32]),
    "stepkv_version": (_I32, []),
    "stepkv_last_cuda_error": (ctypes.c_char_p, []),
    "stepkv_score_workspace_size": (_SZ, [_I32, _I32, _I32, _I32, _I32]),
    "stepkv_score": (_I32, [_I32, _VP, _I64, _VP, _I64, _I32, _I32, _I32, _I32, _I32, _VP, _VP, _SZ, _VP, _VP]),
    "stepkv_score_lse": (_I32, [_I32, _VP, _I64, _VP, _I64, _VP, _I32, _I32, _I32, _I32, _I32, _VP, _VP, _SZ, _VP,
                                _VP]),
    "stepkv_selftest_score_timeout": (_I32, [_I32, _VP, _I64, _VP, _I64, _I32, _I32, _I32, _I32, _I32, _VP, _VP, _SZ,
                                             ctypes.c_uint64, _VP, _VP]),
    "stepkv_select_workspace_size": (_SZ, [_I32, _I32, _I32]),
    "stepkv_select": (_I32, [_VP, _I32, _I32, _VP, _VP, ctypes.POINTER(CSteps), ctypes.POINTER(CParams),
                             ctypes.POINTER(CBudget), ctypes.POINTER(CSelOut), _VP, _SZ, _VP, _VP]),
    "stepkv_select_static_scratch": (_I32, [_VP, _I32, _I32, _VP, _VP, ctypes.POINTER(CSteps),
                                            ctypes.POINTER(CParams), ctypes.POINTER(CBudget),
                                            ctypes.POINTER(CSelOut), _VP, _VP]),
    "stepkv_compact": (_I32, [_I32, _VP, _VP, _I64, _I32, _I32, _I32, _VP, _VP, _I32, _VP, _VP, _I64, _VP, _VP,
                              _VP, _VP, _VP, _VP]),
    "stepkv_decode_workspace_size": (_SZ, [_I32, _I32, _I32, _I32, _I32]),
    "stepkv_decode_h2o_workspace_size": (_SZ, [_I32, _I32, _I32, _I32, _I32]),
    "stepkv_step_signals": (_I32, [_VP, _VP, _I32, _I32, _VP, _VP, _VP, _VP, _VP]),
    "stepkv_set_stage_events": (None, [_VP, _VP, _VP]),
    "stepkv_decode_h2o": (_I32, [_I32, _VP, _VP, _VP, _I64, _I32, _I32, _I32, _VP, _I32, _I32, _VP, _VP, _I64, _VP,
                                 _SZ, _VP, _VP]),
    "stepkv_decode": (_I32, [_I32, _VP, _VP, _VP, _I64, _I32, _I32, _I32, _VP, _I32, _I32, _VP, _VP, _SZ, _VP,
                             _VP]),
    "stepkv_compress_workspace_size": (_SZ, [ctypes.POINTER(CProblem), _I32]),
    "stepkv_compress": (_I32, [ctypes.POINTER(CProblem), _I32, ctypes.POINTER(CParams), _VP, _SZ, _VP, _VP]),
}


def load_library(path: Optional[str] = None):
    """Load libstepkv.so (built in-tree by paper_2609_22158_gb300.build); raises if it is missing."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise StepKVError(STEPKV_ECUDA, "load_library",
                          f"{p} not found: build it with `python -m paper_2609_22158_gb300.build`")
    lib = ctypes.CDLL(p)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    if path is None:
        _lib = lib
    return lib


def status_string(code: int) -> str:
    try:
        return load_library().stepkv_status_string(int(code)).decode()
    except Exception:  # library not built yet
        return "status %d" % code


@dataclass
class Params:
    """Table H defaults (appendix "Implementation Details")."""
    lam: float = 0.3
    w_r: float = 0.85
    w_c: float = 0.15
    r_min: float = -1.0
    r_max: float = 2.0
    s_max: float = 8.0
    eta: float = 1.5
    alpha: float = 0.2
    beta: float = 0.8
    sal_norm: int = NORM_MAX
    sal_pool: int = 1  # SnapKV-style token-axis pooling width (odd; 1 = none), taken by stepkv_select
    sal_pool_mode: int = POOL_MAX

    def c(self) -> CParams:
        return CParams(self.lam, self.w_r, self.w_c, self.r_min, self.r_max, self.s_max, self.eta, self.alpha,
                       self.beta, self.sal_norm, self.sal_pool, self.sal_pool_mode)


def default_params() -> Params:
    cp = CParams()
    load_library().stepkv_default_params(ctypes.byref(cp))
    return Params(cp.lambda_, cp.w_r, cp.w_c, cp.r_min, cp.r_max, cp.s_max, cp.eta, cp.alpha, cp.beta, cp.sal_norm,
                  cp.sal_pool, cp.sal_pool_mode)


# ----------------------------------------------------------------------------- helpers
def _torch():
    import torch
    return torch


def _ptr(t) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream_handle(stream) -> int:
    torch = _torch()
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _check(code: int, where: str):
    if code != STEPKV_OK:
        detail = ""
        if code == STEPKV_ECUDA:
            detail = load_library().stepkv_last_cuda_error().decode()
        raise StepKVError(code, where, detail)


def _need(t, dtype, name, ndim=None, host=False):
    torch = _torch()
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if host:
        if t.is_cuda or not t.is_pinned():
            raise ValueError(f"{name} must be in page-locked host memory (pin_memory())")
    elif not t.is_cuda:
        raise ValueError(f"{name} must be on a CUDA device")
    if ndim is not None and t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dims")
    return t


def _rows_layout(ts: Sequence, name: str, host=False):
    """[H, rows, d] bf16 tensors with unit stride in d and dense rows; returns (head_stride, rows)."""
    torch = _torch()
    hs = None
    for i, t in enumerate(ts):
        _need(t, torch.bfloat16, f"{name}[{i}]", 3, host=host)
        H, R, d = t.shape
        if t.stride(2) != 1 or (R > 1 and t.stride(1) != d):
            raise ValueError(f"{name}[{i}] rows must be dense (stride(1) == d, stride(2) == 1)")
        s = t.stride(0) if H > 1 else R * d
        if hs is None:
            hs = s
        elif hs != s:
            raise ValueError(f"all {name} tensors must share one head stride")
    return hs


def _ptr_array(ts) -> ctypes.Array:
    arr = (ctypes.c_void_p * max(1, len(ts)))()
    for i, t in enumerate(ts):
        arr[i] = t.data_ptr()
    return arr


def new_status(device=None):
    torch = _torch()
    return torch.zeros(1, dtype=torch.int32, device=device or "cuda")


def _workspace(nbytes: int, ws, device):
    torch = _torch()
    if ws is None:
        ws = torch.empty(max(nbytes, 256) + 256, dtype=torch.uint8, device=device)
    if ws.numel() < nbytes:
        raise ValueError(f"workspace too small: {ws.numel()} < {nbytes}")
    return ws


def _aligned_ws(ws):
    off = (-ws.data_ptr()) % 256
    return ws.data_ptr() + off, ws.numel() - off


# ----------------------------------------------------------------------------- stage 1
def stepkv_score(K: Sequence, Q: Sequence, T: int, W: Optional[int] = None, sal=None, ws=None, status=None,
                 stream=None, lse: Optional[Sequence] = None):
    """Window-attention saliency of len(K) layers: returns sal [n_layers, Hkv, T] float32.
    K[l]: [Hkv, rows >= T, d] bf16; Q[l]: [Hq, W, d] bf16 (query w at slot T-W+w).  With lse (per layer
    [Hq, W] float32, each query's natural-log causal log-sum-exp, as a prefill attention reports it) the
    row statistics are taken from it and only the second pass runs (stepkv_score_lse)."""
    torch = _torch()
    lib = load_library()
    n = len(K)
    if n != len(Q) or n == 0:
        raise ValueError("K and Q need the same non-zero number of layers")
    ks = _rows_layout(K, "K")
    qs = _rows_layout(Q, "Q")
    Hkv, _, d = K[0].shape
    Hq, Wq, dq = Q[0].shape
    W = Wq if W is None else W
    if dq != d:
        raise ValueError("K and Q head dims differ")
    dev = K[0].device
    if sal is None:
        sal = torch.empty((n, Hkv, T), dtype=torch.float32, device=dev)
    _need(sal, torch.float32, "sal")
    need = lib.stepkv_score_workspace_size(n, Hkv, Hq, T, W)
    ws = _workspace(need + 256, ws, dev)
    wp, wn = _aligned_ws(ws)
    status = status if status is not None else new_status(dev)
    kp, qp = _ptr_array(K), _ptr_array(Q)
    if lse is None:
        code = lib.stepkv_score(n, ctypes.cast(kp, ctypes.c_void_p), ks, ctypes.cast(qp, ctypes.c_void_p), qs, Hkv, Hq,
                                d, T, W, sal.data_ptr(), wp, wn, status.data_ptr(), _stream_handle(stream))
        _check(code, "stepkv_score")
        return sal
    if len(lse) != n:
        raise ValueError("lse needs one tensor per layer")
    for i, t in enumerate(lse):
        _need(t, torch.float32, f"lse[{i}]", 2)
        if tuple(t.shape) != (Hq, W) or not t.is_contiguous():
            raise ValueError(f"lse[{i}] must be a contiguous [Hq, W] float32 tensor")
    lp = _ptr_array(lse)
    code = lib.stepkv_score_lse(n, ctypes.cast(kp, ctypes.c_void_p), ks, ctypes.cast(qp, ctypes.c_void_p), qs,
                                ctypes.cast(lp, ctypes.c_void_p), Hkv, Hq, d, T, W, sal.data_ptr(), wp, wn,
                                status.data_ptr(), _stream_handle(stream))
    _check(code, "stepkv_score_lse")
    return sal


def stepkv_selftest_score_timeout(K: Sequence, Q: Sequence, T: int, wait_limit_ns: int, status, W=None,
                                  stream=None):
    """Failure-path self-test: the saliency kernel with a second-pass wait that runs out after
    wait_limit_ns; STEPKV_ETIMEOUT lands in `status` (caller-zeroed device int32) and the kernel returns."""
    torch = _torch()
    lib = load_library()
    n = len(K)
    ks = _rows_layout(K, "K")
    qs = _rows_layout(Q, "Q")
    Hkv, _, d = K[0].shape
    Hq, Wq, _ = Q[0].shape
    W = Wq if W is None else W
    dev = K[0].device
    sal = torch.empty((n, Hkv, T), dtype=torch.float32, device=dev)
    ws = _workspace(lib.stepkv_score_workspace_size(n, Hkv, Hq, T, W) + 256, None, dev)
    wp, wn = _aligned_ws(ws)
    kp, qp = _ptr_array(K), _ptr_array(Q)
    code = lib.stepkv_selftest_score_timeout(n, ctypes.cast(kp, ctypes.c_void_p), ks, ctypes.cast(qp, ctypes.c_void_p),
                                             qs, Hkv, Hq, d, T, W, sal.data_ptr(), wp, wn, int(wait_limit_ns),
                                             status.data_ptr(), _stream_handle(stream))
    _check(code, "stepkv_selftest_score_timeout")
    return ws


# ----------------------------------------------------------------------------- stages 2-4
@dataclass
class StepSignals:
    """Per-step trajectory signals (device float32 [n_steps]); see stepkv_steps_t."""
    valid: object
    gain: object
    red: object
    reuse_in: object
    obs_sim: object = None
    reuse_out: object = None

    @property
    def n_steps(self) -> int:
        return int(self.valid.numel())

    def c(self) -> CSteps:
        torch = _torch()
        for nm in ("valid", "gain", "red", "reuse_in"):
            _need(getattr(self, nm), torch.float32, nm, 1)
        return CSteps(self.n_steps, _ptr(self.valid), _ptr(self.gain), _ptr(self.red), _ptr(self.obs_sim),
                      _ptr(self.reuse_in), _ptr(self.reuse_out))


def budget_ratio(num: int, den: int) -> CBudget:
    return CBudget(BUDGET_RATIO, int(num), int(den), 0)


def budget_count(n: int) -> CBudget:
    return CBudget(BUDGET_COUNT, 0, 1, int(n))


@dataclass
class SelectOutputs:
    kept_idx: object
    n_kept: object
    n_budget: object = None
    priority: object = None
    token_sal: object = None
    step_util: object = None
    step_count: object = None
    step_sal_sum: object = None
    step_sal_max: object = None
    step_kept: object = None

    @staticmethod
    def allocate(T: int, n_steps: int, kept_cap: int, device, full: bool = True) -> "SelectOutputs":
        torch = _torch()
        i32, f32 = torch.int32, torch.float32
        o = SelectOutputs(torch.full((max(kept_cap, 1),), -1, dtype=i32, device=device),
                          torch.zeros(1, dtype=i32, device=device))
        if full:
            o.n_budget = torch.zeros(2, dtype=i32, device=device)
            o.priority = torch.empty(T, dtype=f32, device=device)
            o.token_sal = torch.empty(T, dtype=f32, device=device)
            o.step_util = torch.empty(n_steps, dtype=f32, device=device)
            o.step_count = torch.empty(n_steps, dtype=i32, device=device)
            o.step_sal_sum = torch.empty(n_steps, dtype=f32, device=device)
            o.step_sal_max = torch.empty(n_steps, dtype=f32, device=device)
            o.step_kept = torch.empty(n_steps, dtype=i32, device=device)
        o._cap = kept_cap
        return o

    def c(self) -> CSelOut:
        cap = getattr(self, "_cap", self.kept_idx.numel())
        return CSelOut(_ptr(self.kept_idx), cap, _ptr(self.n_kept), _ptr(self.n_budget), _ptr(self.priority),
                       _ptr(self.token_sal), _ptr(self.step_util), _ptr(self.step_count), _ptr(self.step_sal_sum),
                       _ptr(self.step_sal_max), _ptr(self.step_kept))


def stepkv_select(sal, step_id, prot, steps: StepSignals, params: Params, budget: CBudget, out: SelectOutputs,
                  ws=None, status=None, stream=None) -> SelectOutputs:
    """Eqs. 1-5 + top-B over the prunable tokens.  sal: [n_sal, T] (or [..., T]) float32 rows."""
    torch = _torch()
    lib = load_library()
    _need(sal, torch.float32, "sal")
    T = sal.shape[-1]
    n_sal = sal.numel() // T
    if not sal.is_contiguous():
        raise ValueError("sal must be contiguous")
    _need(step_id, torch.int32, "step_id", 1)
    _need(prot, torch.uint8, "prot", 1)
    if step_id.numel() < T or prot.numel() < T:
        raise ValueError("step_id/prot shorter than T")
    dev = sal.device
    need = lib.stepkv_select_workspace_size(n_sal, T, steps.n_steps)
    ws = _workspace(need + 256, ws, dev)
    wp, wn = _aligned_ws(ws)
    status = status if status is not None else new_status(dev)
    cs, cp, co = steps.c(), params.c(), out.c()
    code = lib.stepkv_select(sal.data_ptr(), n_sal, T, step_id.data_ptr(), prot.data_ptr(), ctypes.byref(cs),
                             ctypes.byref(cp), ctypes.byref(budget), ctypes.byref(co), wp, wn, status.data_ptr(),
                             _stream_handle(stream))
    _check(code, "stepkv_select")
    return out


# ----------------------------------------------------------------------------- decode attention
def stepkv_decode(q: Sequence, K: Sequence, V: Sequence, n, out: Optional[Sequence] = None, ws=None, status=None,
                  stream=None):
    """One query token per layer over a (compacted) cache: out[l][g] = softmax(q[l][g] K^T / sqrt(d)) V.

    q[l]: [Hq, d] bf16; K[l], V[l]: [Hkv, rows, d] bf16 (rows >= n); n: an int, or a device int32 tensor
    (e.g. the n_kept of a compaction) read on the device.  Returns the list of [Hq, d] fp32 outputs."""
    torch = _torch()
    lib = load_library()
    L = len(q)
    if L < 1 or len(K) != L or len(V) != L:
        raise ValueError("q, K and V need one tensor per layer")
    hs = _rows_layout(list(K) + list(V), "K/V")
    Hkv, rows, d = K[0].shape
    for i, t in enumerate(q):
        _need(t, torch.bfloat16, f"q[{i}]", 2)
        if not t.is_contiguous():
            raise ValueError(f"q[{i}] must be contiguous")
    Hq = q[0].shape[0]
    dev = q[0].device
    if out is None:
        out = [torch.empty((Hq, d), dtype=torch.float32, device=dev) for _ in range(L)]
    for i, t in enumerate(out):
        _need(t, torch.float32, f"out[{i}]", 2)
    if isinstance(n, int):
        n_dev, n_host = None, n
    else:
        _need(n, torch.int32, "n")
        n_dev, n_host = n, 0
    need = lib.stepkv_decode_workspace_size(L, Hkv, Hq, d, rows)
    ws = _workspace(need + 256, ws, dev)
    wp, wn = _aligned_ws(ws)
    status = status if status is not None else new_status(dev)
    arrs = [_ptr_array(q), _ptr_array(K), _ptr_array(V), _ptr_array(out)]
    cv = lambda a: ctypes.cast(a, ctypes.c_void_p)
    code = lib.stepkv_decode(L, cv(arrs[0]), cv(arrs[1]), cv(arrs[2]), hs, Hkv, Hq, d, _ptr(n_dev), n_host, rows,
                             cv(arrs[3]), wp, wn, status.data_ptr(), _stream_handle(stream))
    _check(code, "stepkv_decode")
    return out


def stepkv_decode_h2o(q: Sequence, K: Sequence, V: Sequence, n, mass: Sequence, out: Optional[Sequence] = None,
                      ws=None, status=None, stream=None):
    """stepkv_decode that also adds each key's group-mean softmax weight to mass[l] ([Hkv, >= rows] fp32,
    accumulated in place): the H2O-style accumulated attention.  Returns the outputs as stepkv_decode."""
    torch = _torch()
    lib = load_library()
    L = len(q)
    if L < 1 or len(K) != L or len(V) != L or len(mass) != L:
        raise ValueError("q, K, V and mass need one tensor per layer")
    hs = _rows_layout(list(K) + list(V), "K/V")
    Hkv, rows, d = K[0].shape
    for i, t in enumerate(q):
        _need(t, torch.bfloat16, f"q[{i}]", 2)
        if not t.is_contiguous():
            raise ValueError(f"q[{i}] must be contiguous")
    for i, t in enumerate(mass):
        _need(t, torch.float32, f"mass[{i}]", 2)
        if t.shape[0] != Hkv or t.shape[1] < rows or t.stride(1) != 1 or t.stride(0) != mass[0].stride(0):
            raise ValueError("mass[l] must be [Hkv, >= rows] float32 with unit column stride and one row stride")
    Hq = q[0].shape[0]
    dev = q[0].device
    if out is None:
        out = [torch.empty((Hq, d), dtype=torch.float32, device=dev) for _ in range(L)]
    for i, t in enumerate(out):
        _need(t, torch.float32, f"out[{i}]", 2)
    if isinstance(n, int):
        n_dev, n_host = None, n
    else:
        _need(n, torch.int32, "n")
        n_dev, n_host = n, 0
    need = lib.stepkv_decode_h2o_workspace_size(L, Hkv, Hq, d, rows)
    ws = _workspace(need + 256, ws, dev)
    wp, wn = _aligned_ws(ws)
    status = status if status is not None else new_status(dev)
    arrs = [_ptr_array(q), _ptr_array(K), _ptr_array(V), _ptr_array(out), _ptr_array(mass)]
    cv = lambda a: ctypes.cast(a, ctypes.c_void_p)
    code = lib.stepkv_decode_h2o(L, cv(arrs[0]), cv(arrs[1]), cv(arrs[2]), hs, Hkv, Hq, d, _ptr(n_dev), n_host, rows,
                                 cv(arrs[3]), cv(arrs[4]), mass[0].stride(0), wp, wn, status.data_ptr(),
                                 _stream_handle(stream))
    _check(code, "stepkv_decode_h2o")
    return out


def stepkv_step_signals(cues, n_cues, k0: Optional[int] = None, gain=None, red=None, obs_sim=None, status=None,
                        stream=None):
    """Sec. 4.1 field signals from evidence cues: cues [n_steps, 3, 64] (int32 or uint32 bits of the sorted cue
    ids of Thought / Action / Observation), n_cues [n_steps, 3] int32.  Writes gain/red for steps >= k0 (default
    the newest) and obs_sim of the newest step against every earlier one; returns (gain, red, obs_sim)."""
    torch = _torch()
    lib = load_library()
    if cues.dim() != 3 or cues.shape[1] != 3 or cues.shape[2] != 64 or cues.element_size() != 4:
        raise ValueError("cues must be [n_steps, 3, 64] 32-bit")
    _need(n_cues, torch.int32, "n_cues", 2)
    if not cues.is_contiguous() or not n_cues.is_contiguous() or n_cues.shape != cues.shape[:2]:
        raise ValueError("cues and n_cues must be contiguous, n_cues [n_steps, 3]")
    n = cues.shape[0]
    k0 = n - 1 if k0 is None else k0
    dev = cues.device
    gain = gain if gain is not None else torch.full((n,), float("nan"), dtype=torch.float32, device=dev)
    red = red if red is not None else torch.full((n,), float("nan"), dtype=torch.float32, device=dev)
    obs_sim = obs_sim if obs_sim is not None else torch.empty(n, dtype=torch.float32, device=dev)
    for t, nm in ((gain, "gain"), (red, "red"), (obs_sim, "obs_sim")):
        _need(t, torch.float32, nm, 1)
    status = status if status is not None else new_status(dev)
    code = lib.stepkv_step_signals(cues.data_ptr(), n_cues.data_ptr(), n, k0, gain.data_ptr(), red.data_ptr(),
                                   obs_sim.data_ptr(), status.data_ptr(), _stream_handle(stream))
    _check(code, "stepkv_step_signals")
    return gain, red, obs_sim


def set_stage_events(before=None, after_select=None, after=None):
    """Events (torch.cuda.Event, created with enable_timing) that later stepkv_compress calls of this thread
    record before their first launch, between selection and compaction, and after their last launch;
    no arguments stop the recording."""
    h = lambda e: None if e is None else ctypes.c_void_p(e.cuda_event)
    load_library().stepkv_set_stage_events(h(before), h(after_select), h(after))


# Limits of the fixed scratch compiled into the library (STEPKV_STATIC_SCRATCH_MAX_* in the header).
STATIC_SCRATCH_MAX_T = 262144
STATIC_SCRATCH_MAX_STEPS = 4096


def stepkv_select_static_scratch(sal, step_id, prot, steps: StepSignals, params: Params, budget: CBudget,
                                 out: SelectOutputs, status, stream=None) -> SelectOutputs:
    """stepkv_select without a workspace, for callers that cannot allocate device memory at call time
    (device memory reserved up front, no room for the synchronisation of a free, no caching allocator).
    The library uses a fixed device scratch instead (T <= 262144, n_steps <= 4096); this wrapper
    allocates nothing either, so `status` (a zeroed device int32) is required.  The first call on a
    device looks up the scratch address and should come before any stream capture; calls that overlap
    on one device share the scratch and race."""
    torch = _torch()
    lib = load_library()
    _need(sal, torch.float32, "sal")
    T = sal.shape[-1]
    n_sal = sal.numel() // T
    if not sal.is_contiguous():
        raise ValueError("sal must be contiguous")
    _need(step_id, torch.int32, "step_id", 1)
    _need(prot, torch.uint8, "prot", 1)
    _need(status, torch.int32, "status")
    if step_id.numel() < T or prot.numel() < T:
        raise ValueError("step_id/prot shorter than T")
    if T > STATIC_SCRATCH_MAX_T or steps.n_steps > STATIC_SCRATCH_MAX_STEPS:
        raise ValueError(f"T={T}, n_steps={steps.n_steps} exceed the static scratch limits "
                         f"({STATIC_SCRATCH_MAX_T}, {STATIC_SCRATCH_MAX_STEPS}): use stepkv_select")
    cs, cp, co = steps.c(), params.c(), out.c()
    code = lib.stepkv_select_static_scratch(sal.data_ptr(), n_sal, T, step_id.data_ptr(), prot.data_ptr(),
                                            ctypes.byref(cs), ctypes.byref(cp), ctypes.byref(budget),
                                            ctypes.byref(co), status.data_ptr(), _stream_handle(stream))
    _check(code, "stepkv_select_static_scratch")
    return out


# ----------------------------------------------------------------------------- stage 5
def stepkv_compact(K_in: Sequence, V_in: Optional[Sequence], T: int, kept_idx, n_kept, kept_cap: int,
                   K_out: Sequence, V_out: Optional[Sequence], step_id_in=None, pos_in=None, step_id_out=None,
                   pos_out=None, status=None, stream=None):
    """Gather retained rows of every layer: K_out[l][h, r] = K_in[l][h, kept_idx[r]] (same for V)."""
    torch = _torch()
    lib = load_library()
    n = len(K_in)
    ins = _rows_layout(K_in + (list(V_in) if V_in else []), "K_in/V_in") if n else 0
    outs = _rows_layout(K_out + (list(V_out) if V_out else []), "K_out/V_out") if n else 0
    Hkv, _, d = K_in[0].shape if n else (1, 0, 8)
    _need(kept_idx, torch.int32, "kept_idx", 1)
    _need(n_kept, torch.int32, "n_kept")
    dev = kept_idx.device
    status = status if status is not None else new_status(dev)
    kin, vin, kout, vout = _ptr_array(K_in), _ptr_array(V_in or []), _ptr_array(K_out), _ptr_array(V_out or [])
    code = lib.stepkv_compact(n, ctypes.cast(kin, ctypes.c_void_p) if n else None,
                              ctypes.cast(vin, ctypes.c_void_p) if V_in else None, ins, Hkv, d, T,
                              kept_idx.data_ptr(), n_kept.data_ptr(), kept_cap,
                              ctypes.cast(kout, ctypes.c_void_p) if n else None,
                              ctypes.cast(vout, ctypes.c_void_p) if V_out else None, outs,
                              _ptr(step_id_in), _ptr(pos_in), _ptr(step_id_out), _ptr(pos_out), status.data_ptr(),
                              _stream_handle(stream))
    _check(code, "stepkv_compact")


# ----------------------------------------------------------------------------- fused pass
@dataclass
class Problem:
    """One trajectory for stepkv_compress (tensors on the device)."""
    K: List            # L x [Hkv, rows >= T, d] bf16
    V: List
    Q: List            # n_sal_layers x [Hq, W, d] bf16 (layers L-n_sal_layers .. L-1)
    T: int
    step_id: object    # [T] int32
    prot: object       # [T] uint8
    steps: StepSignals
    budget: CBudget
    K_out: List
    V_out: List
    out: SelectOutputs
    pos_in: object = None
    step_id_out: object = None
    pos_out: object = None
    # STEPKV_MEM_HOST: K/V (or K_out/V_out) are pinned host tensors that the compaction reads (writes)
    # over the CPU-GPU link; the saliency stage then reads K_sal (device copies of the last
    # n_sal_layers layers' K)
    kv_location: int = STEPKV_MEM_DEVICE
    out_location: int = STEPKV_MEM_DEVICE
    K_sal: Optional[List] = None
    # n_sal_layers x [Hq, W] float32: each window query's natural-log causal log-sum-exp from the
    # Observation prefill; given, the saliency stage runs its second pass only
    sal_lse: Optional[List] = None
    _keep: list = field(default_factory=list, repr=False)
    _c: object = field(default=None, repr=False)

    def c(self) -> CProblem:
        """The C struct, validated and built on first use and reused afterwards (building it checks
        every per-layer tensor, which costs more host time than the pass itself takes on the GPU).
        Call refresh() after replacing or reshaping any tensor of the problem."""
        if self._c is None:
            self._c = self._build()
        return self._c

    def refresh(self):
        self._c = None

    def _build(self) -> CProblem:
        torch = _torch()
        L = len(self.K)
        Ls = len(self.Q)
        kv_host = self.kv_location == STEPKV_MEM_HOST
        ks = _rows_layout(list(self.K) + list(self.V), "K/V", host=kv_host)
        qs = _rows_layout(self.Q, "Q")
        outs = _rows_layout(list(self.K_out) + list(self.V_out), "K_out/V_out",
                            host=self.out_location == STEPKV_MEM_HOST)
        if kv_host:
            if self.K_sal is None or len(self.K_sal) != Ls:
                raise ValueError("a host-resident cache needs K_sal: device copies of the saliency layers' K")
            if _rows_layout(self.K_sal, "K_sal") != ks:
                raise ValueError("K_sal must share the head stride of K")
        Hkv, _, d = self.K[0].shape
        Hq, W, _ = self.Q[0].shape
        _need(self.step_id, torch.int32, "step_id", 1)
        _need(self.prot, torch.uint8, "prot", 1)
        if self.sal_lse is not None:
            if len(self.sal_lse) != Ls:
                raise ValueError("sal_lse needs one [Hq, W] tensor per saliency layer")
            for i, t in enumerate(self.sal_lse):
                _need(t, torch.float32, f"sal_lse[{i}]", 2)
                if tuple(t.shape) != (Hq, W) or not t.is_contiguous():
                    raise ValueError(f"sal_lse[{i}] must be a contiguous [Hq, W] float32 tensor")
        arrs = [_ptr_array(self.K), _ptr_array(self.V), _ptr_array(self.Q), _ptr_array(self.K_out),
                _ptr_array(self.V_out), _ptr_array(self.K_sal or []), _ptr_array(self.sal_lse or [])]
        self._keep = arrs
        cv = lambda a: ctypes.cast(a, ctypes.c_void_p)
        return CProblem(L, Hkv, Hq, d, self.T, W, Ls, cv(arrs[0]), cv(arrs[1]), ks, cv(arrs[2]), qs,
                        _ptr(self.step_id), _ptr(self.prot), _ptr(self.pos_in), self.steps.c(), self.budget,
                        cv(arrs[3]), cv(arrs[4]), outs, _ptr(self.step_id_out), _ptr(self.pos_out), self.out.c(),
                        self.kv_location, self.out_location, cv(arrs[5]) if kv_host else None,
                        cv(arrs[6]) if self.sal_lse is not None else None)


def stepkv_workspace_size(problems: Sequence[Problem]) -> int:
    arr = (CProblem * len(problems))(*[p.c() for p in problems])
    return int(load_library().stepkv_compress_workspace_size(arr, len(problems)))


def stepkv_compress(problems: Sequence[Problem], params: Params, ws=None, status=None, stream=None):
    """score -> reduce/fuse -> select -> compact for every trajectory, in order on one stream."""
    lib = load_library()
    probs = list(problems)
    arr = (CProblem * len(probs))(*[p.c() for p in probs])
    need = int(lib.stepkv_compress_workspace_size(arr, len(probs)))
    dev = probs[0].step_id.device
    ws = _workspace(need + 256, ws, dev)
    wp, wn = _aligned_ws(ws)
    status = status if status is not None else new_status(dev)
    cp = params.c()
    code = lib.stepkv_compress(arr, len(probs), ctypes.byref(cp), wp, wn, status.data_ptr(), _stream_handle(stream))
    _check(code, "stepkv_compress")
    return status
