"""Python binding of libfastvr_attn.so (the C ABI in include/fastvr_attn.h).

The functions below carry the C names and only marshal arguments: pointers are
passed as integers (device addresses), streams as cudaStream_t handles.  Every
step of the computation runs in the library's CUDA kernels; there is no
fallback of any kind, and importing this module raises when the library has
not been built.

`StreamingAttention` is a convenience wrapper for torch tensors: it allocates
the KV cache with torch (device memory is the caller's in the C ABI) and
passes data pointers and the current CUDA stream through.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Tuple

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libfastvr_attn.so")
# The same library with device-side index checks (FASTVR_BOUNDS_CHECK).
DEBUG_LIB_PATH = os.path.join(_HERE, "libfastvr_attn_debug.so")

FASTVR_OK = 0
FASTVR_ERR_INVALID_ARG = 1
FASTVR_ERR_UNSUPPORTED = 2
FASTVR_ERR_CAPACITY = 3
FASTVR_ERR_SEQUENCE = 4
FASTVR_ERR_CUDA = 5
FASTVR_ERR_TIMEOUT = 6
FASTVR_ERR_BOUNDS = 7


class fastvr_attn_config_t(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32),
                ("tokens_per_frame", ctypes.c_int32),
                ("frames_per_chunk", ctypes.c_int32),
                ("window_chunks", ctypes.c_int32),
                ("max_chunks", ctypes.c_int32),
                ("softmax_scale", ctypes.c_float)]


# Every symbol the header declares, with (restype, argtypes).
_VP, _I32, _I64, _SZ = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64,
                        ctypes.c_size_t)
_CFGP = ctypes.POINTER(fastvr_attn_config_t)
SIGNATURES = {
    "fastvr_kv_cache_bytes": (_I32, [_CFGP, ctypes.POINTER(_SZ)]),
    "fastvr_attn_plan": (_I32, [_CFGP, _VP, _SZ, ctypes.POINTER(_VP)]),
    "fastvr_kv_append": (_I32, [_VP, _VP, _VP, _I32, _VP]),
    "fastvr_chunk_attn_fwd": (_I32, [_VP, _VP, _VP, _VP, _VP]),
    "fastvr_plan_reset": (_I32, [_VP]),
    "fastvr_get_status": (_I32, [_VP]),
    "fastvr_plan_get_state": (_I32, [_VP, ctypes.POINTER(_I64),
                                     ctypes.POINTER(_I32)]),
    "fastvr_plan_set_state": (_I32, [_VP, _I64, _I32]),
    "fastvr_plan_visible": (_I32, [_VP, ctypes.POINTER(_I32),
                                   ctypes.POINTER(_I64),
                                   ctypes.POINTER(_I64),
                                   ctypes.POINTER(_I64)]),
    "fastvr_plan_launch_count": (_I32, [_VP, ctypes.POINTER(_I64)]),
    "fastvr_one_step_update": (_I32, [_VP, _VP, _VP, _I64, ctypes.c_float,
                                      _I32, _VP]),
    "fastvr_blockcausal_bwd_scratch_bytes": (_I32, [_CFGP, _I32,
                                                    ctypes.POINTER(_SZ)]),
    "fastvr_blockcausal_attn_bwd": (_I32, [_CFGP, _I32] + [_VP] * 10 +
                                    [_SZ, _VP]),
    "fastvr_blockcausal_attn_fwd": (_I32, [_CFGP, _I32, _VP, _VP, _VP, _VP,
                                           _VP, _VP]),
    "fastvr_chunk_attn_fwd_static": (_I32, [_CFGP, _VP, _I32, _VP, _VP, _I64,
                                            _I32, ctypes.POINTER(_I64),
                                            ctypes.POINTER(_I64), _VP, _VP,
                                            _VP]),
    "fastvr_debug_inject_stall": (_I32, [_VP, _I32, ctypes.c_uint64]),
    "fastvr_debug_shift_next_append": (_I32, [_VP, _I64]),
    "fastvr_get_device_status": (_I32, []),
    "fastvr_debug_inject_stall_noplan": (_I32, [_I32, ctypes.c_uint64]),
    "fastvr_plan_destroy": (None, [_VP]),
    "fastvr_status_string": (ctypes.c_char_p, [_I32]),
}


def _load(path: str = LIB_PATH) -> ctypes.CDLL:
    if not os.path.exists(path):
        raise ImportError(
            f"{path} is missing: build it with "
            "`python -m paper_2609_36757_gb300.build` (there is no fallback)")
    lib = ctypes.CDLL(path)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


lib = _load()


def use_library(path: str) -> ctypes.CDLL:
    """Route every call of this module to the library at path (e.g.
    DEBUG_LIB_PATH) and return the one used before."""
    global lib
    previous, lib = lib, _load(path)
    return previous


class FastVRError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {fastvr_status_string(status)}")


def _check(status: int, where: str) -> None:
    if status != FASTVR_OK:
        raise FastVRError(status, where)


# ------------------------------------------------------------ C-named calls
def fastvr_status_string(status: int) -> str:
    return lib.fastvr_status_string(status).decode()


def fastvr_kv_cache_bytes(cfg: fastvr_attn_config_t) -> int:
    n = _SZ(0)
    _check(lib.fastvr_kv_cache_bytes(ctypes.byref(cfg), ctypes.byref(n)),
           "fastvr_kv_cache_bytes")
    return n.value


def fastvr_attn_plan(cfg: fastvr_attn_config_t, kv_cache: int,
                     nbytes: int) -> int:
    plan = _VP()
    _check(lib.fastvr_attn_plan(ctypes.byref(cfg), kv_cache, nbytes,
                                ctypes.byref(plan)), "fastvr_attn_plan")
    return plan.value


def fastvr_kv_append(plan: int, k_new: int, v_new: int, frames: int,
                     stream: int) -> None:
    _check(lib.fastvr_kv_append(plan, k_new, v_new, frames, stream),
           "fastvr_kv_append")


def fastvr_chunk_attn_fwd(plan: int, q: int, out: int, lse: int,
                          stream: int) -> None:
    _check(lib.fastvr_chunk_attn_fwd(plan, q, out, lse, stream),
           "fastvr_chunk_attn_fwd")


def fastvr_plan_reset(plan: int) -> None:
    _check(lib.fastvr_plan_reset(plan), "fastvr_plan_reset")


def fastvr_get_status(plan: int) -> int:
    return lib.fastvr_get_status(plan)


def fastvr_plan_get_state(plan: int) -> Tuple[int, int]:
    c, f = _I64(0), _I32(0)
    _check(lib.fastvr_plan_get_state(plan, ctypes.byref(c), ctypes.byref(f)),
           "fastvr_plan_get_state")
    return c.value, f.value


def fastvr_plan_set_state(plan: int, chunks: int, last_frames: int) -> None:
    _check(lib.fastvr_plan_set_state(plan, chunks, last_frames),
           "fastvr_plan_set_state")


def fastvr_plan_visible(plan: int):
    """[(start, len), ...] token ranges of a head's cache, and their total."""
    n = _I32(0)
    st, ln = (_I64 * 2)(), (_I64 * 2)()
    tot = _I64(0)
    _check(lib.fastvr_plan_visible(plan, ctypes.byref(n), st, ln,
                                   ctypes.byref(tot)), "fastvr_plan_visible")
    return [(st[i], ln[i]) for i in range(n.value)], tot.value


def fastvr_chunk_attn_fwd_static(cfg: fastvr_attn_config_t, q: int,
                                 q_frames: int, k_cache: int, v_cache: int,
                                 cache_tokens: int, segments, out: int,
                                 lse: int, stream: int) -> None:
    """The allocation-free attention entry point; `segments` is a list of
    (start, len) key ranges of one head's cache."""
    n = len(segments)
    st = (_I64 * max(2, n))(*[s for s, _ in segments])
    ln = (_I64 * max(2, n))(*[l for _, l in segments])
    _check(lib.fastvr_chunk_attn_fwd_static(
        ctypes.byref(cfg), q, q_frames, k_cache, v_cache, cache_tokens, n, st,
        ln, out, lse, stream), "fastvr_chunk_attn_fwd_static")


def fastvr_blockcausal_attn_fwd(cfg: fastvr_attn_config_t, num_frames: int,
                                q: int, k: int, v: int, out: int, lse: int,
                                stream: int) -> None:
    _check(lib.fastvr_blockcausal_attn_fwd(ctypes.byref(cfg), num_frames, q,
                                           k, v, out, lse, stream),
           "fastvr_blockcausal_attn_fwd")


def blockcausal_attention(cfg: fastvr_attn_config_t, q, k, v,
                          want_lse: bool = False):
    """Torch convenience for fastvr_blockcausal_attn_fwd: q, k, v contiguous
    bfloat16 CUDA tensors [B, L, H, d]; runs on the current stream."""
    import torch
    for t in (q, k, v):
        if t.dtype != torch.bfloat16 or not t.is_cuda or not t.is_contiguous():
            raise ValueError("q, k, v must be contiguous bfloat16 CUDA tensors")
    if not (q.shape == k.shape == v.shape):
        raise ValueError("q, k, v differ in shape")
    B, L, H, d = q.shape
    if (B, H, d) != (cfg.batch, cfg.heads, cfg.head_dim) or \
            L % cfg.tokens_per_frame:
        raise ValueError(f"q has shape {tuple(q.shape)}")
    out = torch.empty_like(q)
    lse = (torch.empty((B, H, L), dtype=torch.float32, device=q.device)
           if want_lse else None)
    fastvr_blockcausal_attn_fwd(cfg, L // cfg.tokens_per_frame, q.data_ptr(),
                                k.data_ptr(), v.data_ptr(), out.data_ptr(),
                                0 if lse is None else lse.data_ptr(),
                                torch.cuda.current_stream().cuda_stream)
    return (out, lse) if want_lse else out


def fastvr_blockcausal_bwd_scratch_bytes(cfg: fastvr_attn_config_t,
                                         num_frames: int) -> int:
    n = _SZ(0)
    _check(lib.fastvr_blockcausal_bwd_scratch_bytes(ctypes.byref(cfg),
                                                    num_frames, ctypes.byref(n)),
           "fastvr_blockcausal_bwd_scratch_bytes")
    return n.value


def fastvr_blockcausal_attn_bwd(cfg, num_frames, q, k, v, out, dout, lse, dq,
                                dk, dv, scratch, scratch_bytes, stream) -> None:
    _check(lib.fastvr_blockcausal_attn_bwd(
        ctypes.byref(cfg), num_frames, q, k, v, out, dout, lse, dq, dk, dv,
        scratch, scratch_bytes, stream), "fastvr_blockcausal_attn_bwd")


def blockcausal_attention_bwd(cfg: fastvr_attn_config_t, q, k, v, out, dout,
                              lse):
    """Torch convenience for fastvr_blockcausal_attn_bwd: bfloat16 CUDA
    tensors [B, L, H, d] and the forward's float32 lse [B, H, L]; returns
    (dq, dk, dv).  The scratch is allocated with torch."""
    import torch
    L = q.shape[1]
    frames = L // cfg.tokens_per_frame
    nbytes = fastvr_blockcausal_bwd_scratch_bytes(cfg, frames)
    scratch = torch.empty(nbytes // 4, dtype=torch.float32, device=q.device)
    dq, dk, dv = (torch.empty_like(q) for _ in range(3))
    fastvr_blockcausal_attn_bwd(
        cfg, frames, q.data_ptr(), k.data_ptr(), v.data_ptr(), out.data_ptr(),
        dout.data_ptr(), lse.data_ptr(), dq.data_ptr(), dk.data_ptr(),
        dv.data_ptr(), scratch.data_ptr(), nbytes,
        torch.cuda.current_stream().cuda_stream)
    return dq, dk, dv


def fastvr_one_step_update(z_lq: int, v: int, z_hat: int, n: int,
                           sigma: float, dtype: int, stream: int) -> None:
    _check(lib.fastvr_one_step_update(z_lq, v, z_hat, n, sigma, dtype, stream),
           "fastvr_one_step_update")


def one_step_update(z_lq, v, sigma: float, out=None):
    """Torch convenience: z_lq bfloat16 or float32, v bfloat16, same shape,
    contiguous CUDA tensors; returns z_lq - sigma * v (in place when
    out is z_lq)."""
    import torch
    if v.dtype != torch.bfloat16 or z_lq.dtype not in (torch.bfloat16,
                                                       torch.float32):
        raise ValueError("z_lq must be bfloat16 or float32 and v bfloat16")
    if z_lq.shape != v.shape or not (z_lq.is_contiguous() and v.is_contiguous()):
        raise ValueError("z_lq and v must be contiguous and of one shape")
    if out is None:
        out = torch.empty_like(z_lq)
    fastvr_one_step_update(z_lq.data_ptr(), v.data_ptr(), out.data_ptr(),
                           z_lq.numel(), sigma,
                           0 if z_lq.dtype == torch.bfloat16 else 1,
                           torch.cuda.current_stream().cuda_stream)
    return out


def fastvr_plan_launch_count(plan: int) -> int:
    n = _I64(0)
    _check(lib.fastvr_plan_launch_count(plan, ctypes.byref(n)),
           "fastvr_plan_launch_count")
    return n.value


def fastvr_debug_inject_stall(plan: int, stall: int,
                              wait_limit_ns: int) -> None:
    _check(lib.fastvr_debug_inject_stall(plan, stall, wait_limit_ns),
           "fastvr_debug_inject_stall")


def fastvr_debug_shift_next_append(plan: int, tokens: int) -> None:
    _check(lib.fastvr_debug_shift_next_append(plan, tokens),
           "fastvr_debug_shift_next_append")


def fastvr_get_device_status() -> int:
    """Status of the calls without a plan on the current device (synchronises;
    a recorded failure is cleared once returned)."""
    return lib.fastvr_get_device_status()


def fastvr_debug_inject_stall_noplan(stall: int, wait_limit_ns: int) -> None:
    _check(lib.fastvr_debug_inject_stall_noplan(stall, wait_limit_ns),
           "fastvr_debug_inject_stall_noplan")


def fastvr_plan_destroy(plan: int) -> None:
    lib.fastvr_plan_destroy(plan)


def make_config(batch: int, heads: int, head_dim: int, tokens_per_frame: int,
                frames_per_chunk: int, window_chunks: int = -1,
                max_chunks: int = 0, softmax_scale: float = 0.0
                ) -> fastvr_attn_config_t:
    return fastvr_attn_config_t(batch, heads, head_dim, tokens_per_frame,
                                frames_per_chunk, window_chunks, max_chunks,
                                softmax_scale)


# ------------------------------------------------------- torch convenience
class StreamingAttention:
    """One video stream: a caller-side KV cache tensor plus a plan.

    append(k, v) and forward(q) take bfloat16 CUDA tensors [B, f*N, H, d]
    (contiguous, token-major) and enqueue on the current CUDA stream."""

    def __init__(self, cfg: fastvr_attn_config_t, device=None):
        import torch
        self.cfg = cfg
        self.nbytes = fastvr_kv_cache_bytes(cfg)
        self.cache = torch.empty(self.nbytes, dtype=torch.uint8,
                                 device=device or "cuda")
        self.plan = fastvr_attn_plan(cfg, self.cache.data_ptr(), self.nbytes)

    def __del__(self):
        plan = getattr(self, "plan", None)
        if plan:
            fastvr_plan_destroy(plan)
            self.plan = None

    def _check_chunk(self, t, name: str) -> int:
        import torch
        c = self.cfg
        if t.dtype != torch.bfloat16 or not t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous bfloat16 CUDA tensor")
        B, L, H, d = t.shape
        if (B, H, d) != (c.batch, c.heads, c.head_dim) or L % c.tokens_per_frame:
            raise ValueError(f"{name} has shape {tuple(t.shape)}")
        return L // c.tokens_per_frame

    @staticmethod
    def _stream() -> int:
        import torch
        return torch.cuda.current_stream().cuda_stream

    def append(self, k, v) -> None:
        frames = self._check_chunk(k, "k")
        if self._check_chunk(v, "v") != frames:
            raise ValueError("k and v differ in length")
        fastvr_kv_append(self.plan, k.data_ptr(), v.data_ptr(), frames,
                         self._stream())

    def forward(self, q, out=None, lse: Optional[object] = None,
                want_lse: bool = False):
        import torch
        self._check_chunk(q, "q")
        if out is None:
            out = torch.empty_like(q)
        if lse is None and want_lse:
            B, L, H, _ = q.shape
            lse = torch.empty((B, H, L), dtype=torch.float32, device=q.device)
        fastvr_chunk_attn_fwd(self.plan, q.data_ptr(), out.data_ptr(),
                              0 if lse is None else lse.data_ptr(),
                              self._stream())
        return (out, lse) if want_lse or lse is not None else out

    def reset(self) -> None:
        fastvr_plan_reset(self.plan)

    def launch_count(self) -> int:
        return fastvr_plan_launch_count(self.plan)

    def status(self) -> int:
        return fastvr_get_status(self.plan)

    def visible(self):
        return fastvr_plan_visible(self.plan)

    def state(self) -> Tuple[int, int]:
        return fastvr_plan_get_state(self.plan)

    def set_state(self, chunks: int, last_frames: int) -> None:
        fastvr_plan_set_state(self.plan, chunks, last_frames)


def config_from_workload(w) -> fastvr_attn_config_t:
    return make_config(w.batch, w.heads, w.head_dim, w.tokens_per_frame,
                       w.frames_per_chunk, w.window_chunks,
                       w.max_chunks, w.softmax_scale)
