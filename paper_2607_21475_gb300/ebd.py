"""Thin Python binding of libebd (include/ebd.h): argument marshalling only.

Each function carries the name of the C entry point it calls and takes torch
tensors that already live on the GPU (the eviction calls also take K, V and
the scores as page-locked CPU tensors: the library then reads the scores and
only the kept rows from host memory); it checks shapes, dtypes and
contiguity, passes raw pointers plus sizes, and raises ``EbdError`` on a
non-OK status.  Every step of the hot path runs in the library's CUDA
kernels.  PyTorch supplies device memory and the current stream.

If the compiled library is missing the import of any entry point raises: there
is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass

import torch

from .build import LIB

__all__ = [
    "EbdError", "EbdDesign", "EBD_F32", "EBD_BF16", "EBD_RANGE_BOUND", "EBD_RANGE_EXACT",
    "EBD_DEV_CAPACITY", "EBD_DEV_NONFINITE", "EBD_DEV_TIMEOUT", "EBD_SAMPLING_POISSON",
    "EBD_SAMPLING_SYSTEMATIC", "lib", "lib_path",
    "ebd_status_string", "ebd_abi_version", "ebd_philox_uniforms", "ebd_score_workspace_bytes",
    "ebd_score", "ebd_compute_pi", "ebd_evict_workspace_bytes", "ebd_evict", "ebd_select",
    "ebd_gather", "ebd_decode_workspace_bytes", "ebd_workspace_bytes", "ebd_certified_decode",
    "ebd_certified_decode_static", "ebd_certificate_update", "ebd_append", "ebd_reevict",
    "ebd_gather_queries", "ebd_variance_contributions", "ebd_block_scores",
    "ebd_check_stalled_wait", "design_for",
    "CompactCache",
    "alloc_compact", "ABI_FUNCTIONS",
]

EBD_OK = 0
EBD_F32, EBD_BF16 = 0, 1
EBD_RANGE_BOUND, EBD_RANGE_EXACT = 0, 1
EBD_DEV_CAPACITY, EBD_DEV_NONFINITE, EBD_DEV_TIMEOUT = 0x1, 0x2, 0x4
EBD_SAMPLING_POISSON, EBD_SAMPLING_SYSTEMATIC = 0, 1

# Every symbol include/ebd.h declares.
ABI_FUNCTIONS = (
    "ebd_status_string", "ebd_abi_version", "ebd_philox_uniforms", "ebd_score_workspace_bytes",
    "ebd_score", "ebd_compute_pi", "ebd_evict_workspace_bytes", "ebd_evict", "ebd_select",
    "ebd_gather", "ebd_decode_workspace_bytes", "ebd_workspace_bytes", "ebd_certified_decode",
    "ebd_certified_decode_static", "ebd_certificate_update", "ebd_append", "ebd_reevict",
    "ebd_gather_queries", "ebd_variance_contributions", "ebd_block_scores",
    "ebd_check_stalled_wait",
)


class EbdError(RuntimeError):
    def __init__(self, func: str, code: int, msg: str):
        super().__init__(f"{func} failed: {msg} (status {code})")
        self.code = code


class EbdDesign(ctypes.Structure):
    """Mirror of ``ebd_design`` in include/ebd.h."""
    _fields_ = [
        ("batch", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32), ("group", ctypes.c_int32),
        ("head_dim", ctypes.c_int32), ("n_ctx", ctypes.c_int32), ("layer", ctypes.c_int32),
        ("seed", ctypes.c_uint64), ("n_sink", ctypes.c_int32), ("n_recent", ctypes.c_int32),
        ("k_head", ctypes.c_int32), ("budget_tokens", ctypes.c_int32),
        ("bisect_iters", ctypes.c_int32), ("eps", ctypes.c_float), ("sampling", ctypes.c_int32),
    ]


_LIB = None


def lib_path() -> str:
    return LIB


def lib():
    """Load libebd.so once; raise if it has not been built."""
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB):
            raise RuntimeError(f"{LIB} is not built; run `python -c \"import __graft_entry__ as g; "
                               f"g.build()\"` (no CPU fallback exists)")
        L = ctypes.CDLL(LIB)
        c_void_p, i32, u64, f32, sz = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_uint64,
                                       ctypes.c_float, ctypes.c_size_t)
        P = ctypes.POINTER(EbdDesign)
        sig = {
            "ebd_status_string": (ctypes.c_char_p, [ctypes.c_int]),
            "ebd_abi_version": (i32, []),
            "ebd_philox_uniforms": (ctypes.c_int, [u64, i32, i32, i32, i32, c_void_p, c_void_p]),
            "ebd_score_workspace_bytes": (sz, [i32, i32, i32]),
            "ebd_score": (ctypes.c_int, [ctypes.c_int, i32, i32, i32, i32, i32, c_void_p, c_void_p,
                                         c_void_p, c_void_p, sz, c_void_p]),
            "ebd_compute_pi": (ctypes.c_int, [P, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p]),
            "ebd_evict_workspace_bytes": (sz, [P, i32]),
            "ebd_evict": (ctypes.c_int, [P, ctypes.c_int, c_void_p, c_void_p, c_void_p, c_void_p,
                                         i32, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, i32,
                                         c_void_p, c_void_p, sz, c_void_p]),
            "ebd_select": (ctypes.c_int, [P, c_void_p, c_void_p, c_void_p, c_void_p, i32, c_void_p,
                                          c_void_p]),
            "ebd_gather": (ctypes.c_int, [P, ctypes.c_int, c_void_p, c_void_p, c_void_p, c_void_p,
                                          i32, c_void_p, c_void_p, c_void_p]),
            "ebd_decode_workspace_bytes": (sz, [ctypes.c_int, i32, i32, i32, i32, i32]),
            "ebd_workspace_bytes": (sz, [P, i32]),
            "ebd_certified_decode": (ctypes.c_int, [ctypes.c_int, i32, i32, i32, i32, c_void_p,
                                                    c_void_p, c_void_p, c_void_p, c_void_p, i32,
                                                    f32, f32, ctypes.c_int, c_void_p, c_void_p,
                                                    c_void_p, c_void_p, c_void_p, c_void_p,
                                                    c_void_p, sz, c_void_p]),
            "ebd_certified_decode_static": (ctypes.c_int, [
                ctypes.c_int, i32, i32, i32, i32, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                i32, f32, f32, ctypes.c_int, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                c_void_p, c_void_p]),
            "ebd_certificate_update": (ctypes.c_int, [c_void_p, i32, i32, i32, i32, f32, i32,
                                                      c_void_p, c_void_p, c_void_p, c_void_p]),
            "ebd_append": (ctypes.c_int, [ctypes.c_int, i32, i32, i32, c_void_p, c_void_p,
                                          c_void_p, c_void_p, c_void_p, c_void_p, c_void_p,
                                          c_void_p, i32, c_void_p, c_void_p]),
            "ebd_reevict": (ctypes.c_int, [P, ctypes.c_int, c_void_p, c_void_p, c_void_p, c_void_p,
                                           c_void_p, c_void_p, i32, c_void_p, c_void_p, c_void_p,
                                           c_void_p, c_void_p, i32, c_void_p, c_void_p]),
            "ebd_gather_queries": (ctypes.c_int, [ctypes.c_int, i32, i32, i32, i32, i32, c_void_p,
                                                  c_void_p, i32, c_void_p, c_void_p]),
            "ebd_variance_contributions": (ctypes.c_int, [ctypes.c_int, i32, i32, i32, i32,
                                                          c_void_p, c_void_p, c_void_p, c_void_p,
                                                          c_void_p, i32, c_void_p, c_void_p,
                                                          c_void_p, c_void_p]),
            "ebd_block_scores": (ctypes.c_int, [i32, i32, i32, c_void_p, c_void_p, c_void_p, i32,
                                                i32, i32, c_void_p, c_void_p]),
            "ebd_check_stalled_wait": (ctypes.c_int, [c_void_p, c_void_p]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _LIB = L
    return _LIB


# ----------------------------------------------------------------- helpers
def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return EBD_F32
    if t.dtype == torch.bfloat16:
        return EBD_BF16
    raise TypeError(f"unsupported dtype {t.dtype}; expected float32 or bfloat16")


def _ptr(t, dtype=None, shape=None, name="tensor", host_ok=False):
    """Address of a contiguous tensor.  host_ok: a page-locked CPU tensor is
    accepted too (the library reads it from the device over the host link)."""
    if t is None:
        return None
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if not t.is_cuda and not (host_ok and t.is_pinned()):
        raise ValueError(f"{name} must be a CUDA tensor" +
                         (" or a page-locked CPU tensor" if host_ok else ""))
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} has dtype {t.dtype}, expected {dtype}")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _check(name, code):
    if code != EBD_OK:
        raise EbdError(name, code, ebd_status_string(code))


def _workspace(nbytes, device, ws):
    if nbytes == 0:
        return None, 0
    if ws is None:
        ws = torch.empty(nbytes, dtype=torch.uint8, device=device)
    if ws.numel() * ws.element_size() < nbytes:
        raise ValueError(f"workspace too small: {ws.numel() * ws.element_size()} < {nbytes}")
    return ctypes.c_void_p(ws.data_ptr()), ws.numel() * ws.element_size()


# ---------------------------------------------------------------- entry points
def ebd_status_string(code: int) -> str:
    return lib().ebd_status_string(int(code)).decode()


def ebd_abi_version() -> int:
    return int(lib().ebd_abi_version())


def ebd_check_stalled_wait(dev_status: torch.Tensor, stream=None) -> torch.Tensor:
    """Run the bounded-wait failure path: ~2 s later EBD_DEV_TIMEOUT is OR-ed
    into dev_status (int32 CUDA tensor [1]) and the context stays usable."""
    _check("ebd_check_stalled_wait", lib().ebd_check_stalled_wait(
        _ptr(dev_status, torch.int32, (1,), "dev_status"), _stream(stream)))
    return dev_status


def ebd_philox_uniforms(seed: int, layer: int, x0: torch.Tensor, stream=None):
    """x0: int32 CUDA tensor [B, Hkv, N], filled with the uint32 Philox words."""
    B, H, N = x0.shape
    _check("ebd_philox_uniforms", lib().ebd_philox_uniforms(
        int(seed), int(layer), B, H, N, _ptr(x0, torch.int32, name="x0"), _stream(stream)))
    return x0


def ebd_score_workspace_bytes(batch, n_kv_heads, n_obs) -> int:
    return int(lib().ebd_score_workspace_bytes(batch, n_kv_heads, n_obs))


def ebd_score(q_obs: torch.Tensor, K: torch.Tensor, scores: torch.Tensor, workspace=None,
              stream=None):
    B, H, N, d = K.shape
    R = q_obs.shape[2]
    dt = _dtype_code(K)
    ws, wsb = _workspace(ebd_score_workspace_bytes(B, H, R), K.device, workspace)
    _check("ebd_score", lib().ebd_score(
        dt, B, H, d, N, R, _ptr(q_obs, K.dtype, (B, H, R, d), "q_obs"), _ptr(K, name="K"),
        _ptr(scores, torch.float32, (B, H, N), "scores"), ws, wsb, _stream(stream)))
    return scores


def design_for(*, batch, n_kv_heads, group, head_dim, n_ctx, layer=0, seed=0, n_sink=4,
               n_recent=32, k_head, budget_tokens, bisect_iters=40, eps=1e-6,
               sampling=0) -> EbdDesign:
    return EbdDesign(batch, n_kv_heads, group, head_dim, n_ctx, layer, seed, n_sink, n_recent,
                     k_head, budget_tokens, bisect_iters, eps, sampling)


def ebd_compute_pi(design: EbdDesign, scores: torch.Tensor, pi: torch.Tensor,
                   certain_mask=None, dev_status=None, stream=None):
    shp = (design.batch, design.n_kv_heads, design.n_ctx)
    _check("ebd_compute_pi", lib().ebd_compute_pi(
        ctypes.byref(design), _ptr(scores, torch.float32, shp, "scores", True),
        _ptr(pi, torch.float32, shp, "pi"), _ptr(certain_mask, torch.uint8, shp, "certain_mask"),
        _ptr(dev_status, torch.int32, (1,), "dev_status"), _stream(stream)))
    return pi


def ebd_evict_workspace_bytes(design: EbdDesign, n_obs: int) -> int:
    return int(lib().ebd_evict_workspace_bytes(ctypes.byref(design), int(n_obs)))


def ebd_workspace_bytes(design: EbdDesign, capacity: int) -> int:
    """One workspace size serving every call of a layer with this design."""
    return int(lib().ebd_workspace_bytes(ctypes.byref(design), int(capacity)))


@dataclass
class CompactCache:
    K_c: torch.Tensor      # [B, Hkv, cap, d]
    V_c: torch.Tensor      # [B, Hkv, cap, d]
    logw_c: torch.Tensor   # [B, Hkv, cap] float32
    idx_c: torch.Tensor    # [B, Hkv, cap] int32
    n_kept: torch.Tensor   # [B, Hkv] int32
    dev_status: torch.Tensor  # [1] int32

    @property
    def capacity(self) -> int:
        return self.K_c.shape[2]


def alloc_compact(batch, n_kv_heads, capacity, head_dim, dtype, device) -> CompactCache:
    """Caller-side allocation of the compact-cache buffers (plain torch.empty)."""
    return CompactCache(
        torch.empty((batch, n_kv_heads, capacity, head_dim), dtype=dtype, device=device),
        torch.empty((batch, n_kv_heads, capacity, head_dim), dtype=dtype, device=device),
        torch.empty((batch, n_kv_heads, capacity), dtype=torch.float32, device=device),
        torch.empty((batch, n_kv_heads, capacity), dtype=torch.int32, device=device),
        torch.empty((batch, n_kv_heads), dtype=torch.int32, device=device),
        torch.zeros((1,), dtype=torch.int32, device=device),
    )


def ebd_evict(design: EbdDesign, K: torch.Tensor, V: torch.Tensor, scores, q_obs,
              out: CompactCache, workspace=None, stream=None) -> CompactCache:
    B, H, N, d = design.batch, design.n_kv_heads, design.n_ctx, design.head_dim
    dt = _dtype_code(K)
    cap = out.capacity
    n_obs = 0 if q_obs is None else q_obs.shape[2]
    if scores is None and q_obs is None:
        raise ValueError("ebd_evict needs scores or q_obs")
    ws, wsb = (None, 0)
    if scores is None:
        ws, wsb = _workspace(ebd_evict_workspace_bytes(design, n_obs), K.device, workspace)
    host_ok = scores is not None  # K, V, scores may stay in page-locked host memory
    _check("ebd_evict", lib().ebd_evict(
        ctypes.byref(design), dt, _ptr(K, K.dtype, (B, H, N, d), "K", host_ok),
        _ptr(V, K.dtype, (B, H, N, d), "V", True),
        _ptr(scores, torch.float32, (B, H, N), "scores", True),
        _ptr(q_obs, K.dtype, None if q_obs is None else (B, H, n_obs, d), "q_obs"), n_obs,
        _ptr(out.K_c, K.dtype, (B, H, cap, d), "K_c"), _ptr(out.V_c, K.dtype, (B, H, cap, d), "V_c"),
        _ptr(out.logw_c, torch.float32, (B, H, cap), "logw_c"),
        _ptr(out.idx_c, torch.int32, (B, H, cap), "idx_c"),
        _ptr(out.n_kept, torch.int32, (B, H), "n_kept"), cap,
        _ptr(out.dev_status, torch.int32, (1,), "dev_status"), ws, wsb, _stream(stream)))
    return out


def ebd_select(design: EbdDesign, scores: torch.Tensor, out: CompactCache, stream=None):
    """Certainty set, pi, Poisson draw and index compaction (no row copy)."""
    B, H, N = design.batch, design.n_kv_heads, design.n_ctx
    cap = out.capacity
    _check("ebd_select", lib().ebd_select(
        ctypes.byref(design), _ptr(scores, torch.float32, (B, H, N), "scores", True),
        _ptr(out.idx_c, torch.int32, (B, H, cap), "idx_c"),
        _ptr(out.logw_c, torch.float32, (B, H, cap), "logw_c"),
        _ptr(out.n_kept, torch.int32, (B, H), "n_kept"), cap,
        _ptr(out.dev_status, torch.int32, (1,), "dev_status"), _stream(stream)))
    return out


def ebd_gather(design: EbdDesign, K: torch.Tensor, V: torch.Tensor, out: CompactCache,
               stream=None):
    """Copy the kept K/V rows named by out.idx_c into out.K_c / out.V_c."""
    B, H, N, d = design.batch, design.n_kv_heads, design.n_ctx, design.head_dim
    cap = out.capacity
    _check("ebd_gather", lib().ebd_gather(
        ctypes.byref(design), _dtype_code(K), _ptr(K, K.dtype, (B, H, N, d), "K", True),
        _ptr(V, K.dtype, (B, H, N, d), "V", True),
        _ptr(out.idx_c, torch.int32, (B, H, cap), "idx_c"),
        _ptr(out.n_kept, torch.int32, (B, H), "n_kept"), cap,
        _ptr(out.K_c, K.dtype, (B, H, cap, d), "K_c"), _ptr(out.V_c, K.dtype, (B, H, cap, d), "V_c"),
        _stream(stream)))
    return out


def ebd_decode_workspace_bytes(dtype_code, batch, n_kv_heads, group, head_dim, capacity) -> int:
    return int(lib().ebd_decode_workspace_bytes(dtype_code, batch, n_kv_heads, group, head_dim,
                                                capacity))


def ebd_certified_decode(Q: torch.Tensor, K_c: torch.Tensor, V_c: torch.Tensor,
                         logw_c: torch.Tensor, n_kept: torch.Tensor, y: torch.Tensor,
                         lse: torch.Tensor, var_hat: torch.Tensor, b_t: torch.Tensor,
                         radius: torch.Tensor, delta: float = 0.1, eps0: float = 1e-9,
                         range_mode: int = EBD_RANGE_BOUND, dev_status=None, workspace=None,
                         stream=None):
    B, H, cap, d = K_c.shape
    Hq = Q.shape[1]
    if Hq % H:
        raise ValueError("query heads must be a multiple of KV heads")
    G = Hq // H
    dt = _dtype_code(K_c)
    ws, wsb = _workspace(ebd_decode_workspace_bytes(dt, B, H, G, d, cap), K_c.device, workspace)
    f = torch.float32
    _check("ebd_certified_decode", lib().ebd_certified_decode(
        dt, B, H, G, d, _ptr(Q, K_c.dtype, (B, Hq, d), "Q"), _ptr(K_c, name="K_c"),
        _ptr(V_c, K_c.dtype, (B, H, cap, d), "V_c"), _ptr(logw_c, f, (B, H, cap), "logw_c"),
        _ptr(n_kept, torch.int32, (B, H), "n_kept"), cap, float(delta), float(eps0),
        int(range_mode), _ptr(y, f, (B, Hq, d), "y"), _ptr(lse, f, (B, Hq), "lse"),
        _ptr(var_hat, f, (B, Hq), "var_hat"), _ptr(b_t, f, (B, Hq), "b_t"),
        _ptr(radius, f, (B, Hq), "radius"), _ptr(dev_status, torch.int32, (1,), "dev_status"),
        ws, wsb, _stream(stream)))
    return y, lse, var_hat, b_t, radius


def ebd_certified_decode_static(Q: torch.Tensor, K_c: torch.Tensor, V_c: torch.Tensor,
                                logw_c: torch.Tensor, n_kept: torch.Tensor, y: torch.Tensor,
                                lse: torch.Tensor, var_hat: torch.Tensor, b_t: torch.Tensor,
                                radius: torch.Tensor, delta: float = 0.1, eps0: float = 1e-9,
                                range_mode: int = EBD_RANGE_BOUND, dev_status=None, stream=None):
    """ebd_certified_decode without a workspace: for callers that cannot allocate
    device memory, the library uses its own fixed 16 MiB scratch array."""
    B, H, cap, d = K_c.shape
    Hq = Q.shape[1]
    if Hq % H:
        raise ValueError("query heads must be a multiple of KV heads")
    G = Hq // H
    f = torch.float32
    _check("ebd_certified_decode_static", lib().ebd_certified_decode_static(
        _dtype_code(K_c), B, H, G, d, _ptr(Q, K_c.dtype, (B, Hq, d), "Q"), _ptr(K_c, name="K_c"),
        _ptr(V_c, K_c.dtype, (B, H, cap, d), "V_c"), _ptr(logw_c, f, (B, H, cap), "logw_c"),
        _ptr(n_kept, torch.int32, (B, H), "n_kept"), cap, float(delta), float(eps0),
        int(range_mode), _ptr(y, f, (B, Hq, d), "y"), _ptr(lse, f, (B, Hq), "lse"),
        _ptr(var_hat, f, (B, Hq), "var_hat"), _ptr(b_t, f, (B, Hq), "b_t"),
        _ptr(radius, f, (B, Hq), "radius"), _ptr(dev_status, torch.int32, (1,), "dev_status"),
        _stream(stream)))
    return y, lse, var_hat, b_t, radius


def ebd_certificate_update(radius: torch.Tensor, cert: torch.Tensor, first_step: bool,
                           head_stride: int = 4, tau: float = 1.0, step_mean=None, red_flag=None,
                           stream=None):
    """One probed decode step of the deployed certificate: radius [L, B, Hq]
    (this step's r_t of every layer) -> cert [B] = max over probed steps of the
    mean over layers and every `head_stride`-th head; red_flag [B] = cert >= tau."""
    L, B, Hq = radius.shape
    f = torch.float32
    _check("ebd_certificate_update", lib().ebd_certificate_update(
        _ptr(radius, f, (L, B, Hq), "radius"), L, B, Hq, int(head_stride), float(tau),
        1 if first_step else 0, _ptr(step_mean, f, (B,), "step_mean"), _ptr(cert, f, (B,), "cert"),
        _ptr(red_flag, torch.int32, (B,), "red_flag"), _stream(stream)))
    return cert


def ebd_append(cc: "CompactCache", k_new: torch.Tensor, v_new: torch.Tensor,
               positions: torch.Tensor, stream=None) -> "CompactCache":
    """Append one token per unit (pi = 1) to the compact cache `cc` in place.
    k_new, v_new: [B, Hkv, d]; positions: [B] int32 token positions."""
    B, H, cap, d = cc.K_c.shape
    dt = _dtype_code(cc.K_c)
    _check("ebd_append", lib().ebd_append(
        dt, B, H, d, _ptr(k_new, cc.K_c.dtype, (B, H, d), "k_new"),
        _ptr(v_new, cc.K_c.dtype, (B, H, d), "v_new"), _ptr(positions, torch.int32, (B,), "positions"),
        _ptr(cc.K_c, name="K_c"), _ptr(cc.V_c, cc.K_c.dtype, (B, H, cap, d), "V_c"),
        _ptr(cc.logw_c, torch.float32, (B, H, cap), "logw_c"),
        _ptr(cc.idx_c, torch.int32, (B, H, cap), "idx_c"),
        _ptr(cc.n_kept, torch.int32, (B, H), "n_kept"), cap,
        _ptr(cc.dev_status, torch.int32, (1,), "dev_status"), _stream(stream)))
    return cc


def ebd_reevict(design: EbdDesign, scores: torch.Tensor, cc_in: "CompactCache",
                out: "CompactCache", stream=None) -> "CompactCache":
    """Evict the resident cache `cc_in` again into `out` (distinct buffers):
    scores [B, Hkv, cap_in] for the resident rows; design.n_ctx == cap_in."""
    B, H, cap_in, d = cc_in.K_c.shape
    cap_out = out.K_c.shape[2]
    dt = _dtype_code(cc_in.K_c)
    f = torch.float32
    _check("ebd_reevict", lib().ebd_reevict(
        ctypes.byref(design), dt, _ptr(scores, f, (B, H, cap_in), "scores"),
        _ptr(cc_in.K_c, name="K_in"), _ptr(cc_in.V_c, cc_in.K_c.dtype, (B, H, cap_in, d), "V_in"),
        _ptr(cc_in.logw_c, f, (B, H, cap_in), "logw_in"),
        _ptr(cc_in.idx_c, torch.int32, (B, H, cap_in), "idx_in"),
        _ptr(cc_in.n_kept, torch.int32, (B, H), "n_kept_in"), cap_in,
        _ptr(out.K_c, cc_in.K_c.dtype, (B, H, cap_out, d), "K_out"),
        _ptr(out.V_c, cc_in.K_c.dtype, (B, H, cap_out, d), "V_out"),
        _ptr(out.logw_c, f, (B, H, cap_out), "logw_out"),
        _ptr(out.idx_c, torch.int32, (B, H, cap_out), "idx_out"),
        _ptr(out.n_kept, torch.int32, (B, H), "n_kept_out"), cap_out,
        _ptr(out.dev_status, torch.int32, (1,), "dev_status"), _stream(stream)))
    return out


def ebd_gather_queries(Q: torch.Tensor, positions: torch.Tensor, n_kv_heads: int,
                       q_obs=None, stream=None) -> torch.Tensor:
    """Observation rows for ebd_score from prefill queries Q [B, Hq, Nq, d] at
    positions [P] (int32, device): q_obs [B, Hkv, G*P, d], row g*P + p."""
    B, Hq, Nq, d = Q.shape
    if Hq % n_kv_heads:
        raise ValueError("query heads must be a multiple of KV heads")
    G = Hq // n_kv_heads
    P = positions.shape[0]
    if q_obs is None:
        q_obs = torch.empty((B, n_kv_heads, G * P, d), dtype=Q.dtype, device=Q.device)
    _check("ebd_gather_queries", lib().ebd_gather_queries(
        _dtype_code(Q), B, n_kv_heads, G, d, Nq, _ptr(Q, name="Q"),
        _ptr(positions, torch.int32, (P,), "positions"), P,
        _ptr(q_obs, Q.dtype, (B, n_kv_heads, G * P, d), "q_obs"), _stream(stream)))
    return q_obs


def ebd_variance_contributions(Q: torch.Tensor, K_c: torch.Tensor, V_c: torch.Tensor,
                               logw_c: torch.Tensor, n_kept: torch.Tensor, y: torch.Tensor,
                               lse: torch.Tensor, contrib=None, stream=None) -> torch.Tensor:
    """Theorem 2's per-token terms [B, Hq, cap] (they sum to V_hat per head)."""
    B, H, cap, d = K_c.shape
    Hq = Q.shape[1]
    G = Hq // H
    f = torch.float32
    if contrib is None:
        contrib = torch.empty((B, Hq, cap), dtype=f, device=K_c.device)
    _check("ebd_variance_contributions", lib().ebd_variance_contributions(
        _dtype_code(K_c), B, H, G, d, _ptr(Q, K_c.dtype, (B, Hq, d), "Q"), _ptr(K_c, name="K_c"),
        _ptr(V_c, K_c.dtype, (B, H, cap, d), "V_c"), _ptr(logw_c, f, (B, H, cap), "logw_c"),
        _ptr(n_kept, torch.int32, (B, H), "n_kept"), cap, _ptr(y, f, (B, Hq, d), "y"),
        _ptr(lse, f, (B, Hq), "lse"), _ptr(contrib, f, (B, Hq, cap), "contrib"), _stream(stream)))
    return contrib


def ebd_block_scores(contrib: torch.Tensor, idx_c: torch.Tensor, n_kept: torch.Tensor,
                     block: int, n_blocks: int, out=None, stream=None) -> torch.Tensor:
    """Sum of retained contributions per block of `block` original positions."""
    B, H, cap = idx_c.shape
    Hq = contrib.shape[1]
    G = Hq // H
    if out is None:
        out = torch.empty((B, H, n_blocks), dtype=torch.float32, device=idx_c.device)
    _check("ebd_block_scores", lib().ebd_block_scores(
        B, H, G, _ptr(contrib, torch.float32, (B, Hq, cap), "contrib"),
        _ptr(idx_c, torch.int32, (B, H, cap), "idx_c"), _ptr(n_kept, torch.int32, (B, H), "n_kept"),
        cap, int(block), int(n_blocks), _ptr(out, torch.float32, (B, H, n_blocks), "out"),
        _stream(stream)))
    return out
