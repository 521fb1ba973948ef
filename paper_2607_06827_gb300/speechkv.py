"""Python binding of libspeechkv (the C ABI in include/speechkv.h).

Argument marshalling only: tensors are passed as raw device pointers, every
step runs in the library's CUDA kernels, and there is no CPU fallback -- if
the library is missing or was built for another machine, loading raises.
Function names and argument order follow the C entry points.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libspeechkv.so")

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_CAPACITY, ERR_TIMEOUT, ERR_WORKSPACE = range(7)
F32, BF16 = 0, 1
OVERLAP_PRIOR = 1  # SPEECHKV_OVERLAP_PRIOR
MAX_BATCH = 512

# Every function the header declares: name -> (restype, argtypes)
_P = ctypes.c_void_p
_I32, _I64, _F, _SZ = ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
SIGNATURES = {
    "speechkv_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "speechkv_compressed_len": (_I64, [_I32] * 7),
    "speechkv_pool": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _P,
                                     _I32, _I64, _I32, _I32, _I32, _I32, _I32,
                                     ctypes.c_int, _P]),
    "speechkv_append": (ctypes.c_int, [_P, _P, _P, _P, _P, _P,
                                       _I32, _I32, _I32, _I32, _I32, _I32,
                                       ctypes.c_int, _P]),
    "speechkv_decode_workspace_size": (_SZ, [_I32] * 5),
    "speechkv_decode_attn": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _F,
                                            _I32, _I32, _I32, _I32, _I32, _I32,
                                            _I32, _I32, _P, _SZ, ctypes.c_int,
                                            ctypes.c_uint32, _P]),
    "speechkv_decode_step": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, _P, _F,
                                            _I32, _I32, _I32, _I32, _I32, _I32,
                                            _I32, _I32, _P, _SZ, ctypes.c_int,
                                            ctypes.c_uint32, _P]),
    "speechkv_decode_step_noalloc": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, _P, _F,
                                                    _I32, _I32, _I32, _I32, _I32, _I32,
                                                    _I32, _I32, ctypes.c_int,
                                                    ctypes.c_uint32, _P]),
    "speechkv_pool_paged": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _I32, _I32,
                                           _I64, _P, _I32, _I64, _I32, _I32, _I32, _I32, _I32,
                                           ctypes.c_int, _P]),
    "speechkv_append_paged": (ctypes.c_int, [_P, _P, _P, _P, _P, _I32, _I32, _I64, _P, _I32,
                                             _I32, _I32, _I32, _I32, _I32, ctypes.c_int, _P]),
    "speechkv_decode_step_paged": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _I32, _I32, _I64, _P,
                                                  _P, _F, _I32, _I32, _I32, _I32, _I32, _I32,
                                                  _I32, _I32, _P, _SZ, ctypes.c_int,
                                                  ctypes.c_uint32, _P]),
    "speechkv_pool_hidden": (ctypes.c_int, [_P, _P, _P, _P, _P, _P, _P, _P, _P, _I32, _I64,
                                            _I64, _I32, _I32, ctypes.c_int, _P]),
    "speechkv_prefill_attn": (ctypes.c_int, [_P, _P, _I64, _P, _P, _P, _P, _P, _P, _I64, _P, _F,
                                             _I32, _I32, _I32, _I32, _I32, _I32, _I32,
                                             ctypes.c_int, _P]),
    "speechkv_prefill_attn_paged": (ctypes.c_int, [_P, _P, _I64, _P, _P, _P, _P, _P, _P, _I32,
                                                   _I32, _I64, _P, _F, _I32, _I32, _I32, _I32,
                                                   _I32, _I32, _I32, ctypes.c_int, _P]),
    "speechkv_check_device_error": (ctypes.c_int, [_P]),
    "speechkv_selftest_timeout": (ctypes.c_int, [_P]),
}

_lock = threading.Lock()
_lib = None


class SpeechKVError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} ({status})")


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load libspeechkv.so (built by ``paper_2607_06827_gb300.build``)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(path):
            raise RuntimeError(
                f"{path} is missing: build it with paper_2607_06827_gb300.build.build() "
                "(there is no fallback implementation)")
        lib = ctypes.CDLL(path)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype, fn.argtypes = res, args
        _lib = lib
        return lib


def status_string(status: int) -> str:
    return load().speechkv_status_string(status).decode()


def _check(status: int, where: str):
    if status != OK:
        raise SpeechKVError(status, where)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise TypeError(f"unsupported dtype {t.dtype}")


def _ptr(t: torch.Tensor | None):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


def compressed_len(P: int, T: int, N: int, G: int, w: int, layer: int, l0: int) -> int:
    return load().speechkv_compressed_len(P, T, N, G, w, layer, l0)


def pool(k_full, v_full, full_off, P, T, N, gate, k_cache, v_cache, cache_off, length,
         w: int, layer: int, l0: int, stream=None):
    """speechkv_pool: k_full/v_full [full_rows, H_kv, d]; full_off/cache_off
    int64 [B+1]; P/T/N/length int32 [B]; gate fp32 [H_kv, d]."""
    B = length.numel()
    full_rows, H_kv, d = k_full.shape
    _check(load().speechkv_pool(
        _ptr(k_full), _ptr(v_full), _ptr(full_off), _ptr(P), _ptr(T), _ptr(N),
        _ptr(gate), _ptr(k_cache), _ptr(v_cache), _ptr(cache_off), _ptr(length),
        B, full_rows, H_kv, d, w, layer, l0, _dtype_code(k_full), _stream(stream)),
        "speechkv_pool")


def append(k_new, v_new, k_cache, v_cache, cache_off, length, w: int, layer: int, l0: int,
           stream=None):
    """speechkv_append: k_new/v_new [B, H_kv, d]; length int32 [B] (in/out)."""
    B, H_kv, d = k_new.shape
    _check(load().speechkv_append(
        _ptr(k_new), _ptr(v_new), _ptr(k_cache), _ptr(v_cache), _ptr(cache_off),
        _ptr(length), B, H_kv, d, w, layer, l0, _dtype_code(k_new), _stream(stream)),
        "speechkv_append")


def decode_workspace_size(B: int, H_q: int, H_kv: int, d: int, grid_ctas: int = 0) -> int:
    n = load().speechkv_decode_workspace_size(B, H_q, H_kv, d, grid_ctas)
    if n == 0:
        raise SpeechKVError(ERR_INVALID_ARG, "speechkv_decode_workspace_size")
    return n


def new_workspace(B: int, H_q: int, H_kv: int, d: int, grid_ctas: int = 0,
                  device=None) -> torch.Tensor:
    """A zero-filled workspace of the size speechkv_decode_attn needs."""
    n = decode_workspace_size(B, H_q, H_kv, d, grid_ctas)
    return torch.zeros((n + 15) // 16 * 16, dtype=torch.uint8, device=device or "cuda")


def decode_attn(q, k_cache, v_cache, cache_off, length, out, workspace, w: int, layer: int,
                l0: int, H_kv: int, scale: float = 0.0, grid_ctas: int = 0, flags: int = 0,
                stream=None):
    """speechkv_decode_attn: q/out [B, H_q, d]; caches in the head-major
    per-request layout; length int32 [B]."""
    B, H_q, d = q.shape
    _check(load().speechkv_decode_attn(
        _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(cache_off), _ptr(length), _ptr(out),
        float(scale), B, H_q, H_kv, d, w, layer, l0, grid_ctas, _ptr(workspace),
        workspace.numel() * workspace.element_size(), _dtype_code(q), flags, _stream(stream)),
        "speechkv_decode_attn")


def decode_step(q, k_new, v_new, k_cache, v_cache, cache_off, length, out, workspace, w: int,
                layer: int, l0: int, scale: float = 0.0, grid_ctas: int = 0, flags: int = 0,
                stream=None):
    """speechkv_decode_step: append k_new/v_new ([B, H_kv, d]) to the caches
    and attend (q/out [B, H_q, d]) in one launch; length int32 [B] advances."""
    B, H_q, d = q.shape
    H_kv = k_new.shape[1]
    _check(load().speechkv_decode_step(
        _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_cache), _ptr(v_cache), _ptr(cache_off),
        _ptr(length), _ptr(out), float(scale), B, H_q, H_kv, d, w, layer, l0, grid_ctas,
        _ptr(workspace), workspace.numel() * workspace.element_size(), _dtype_code(q), flags,
        _stream(stream)),
        "speechkv_decode_step")


def decode_step_noalloc(q, k_new, v_new, k_cache, v_cache, cache_off, length, out, w: int,
                        layer: int, l0: int, scale: float = 0.0, grid_ctas: int = 0,
                        flags: int = 0, stream=None):
    """speechkv_decode_step_noalloc: decode_step for callers that may not
    allocate device memory; the library's own fixed scratch replaces the
    workspace (see include/speechkv.h for its size limit and sharing rules)."""
    B, H_q, d = q.shape
    H_kv = k_new.shape[1]
    _check(load().speechkv_decode_step_noalloc(
        _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_cache), _ptr(v_cache), _ptr(cache_off),
        _ptr(length), _ptr(out), float(scale), B, H_q, H_kv, d, w, layer, l0, grid_ctas,
        _dtype_code(q), flags, _stream(stream)),
        "speechkv_decode_step_noalloc")


def _pages(k_pages, block_table):
    """(num_blocks, block_size) of pages shaped [num_blocks, H_kv, block_size, d]."""
    if k_pages.dim() != 4:
        raise ValueError("pages must be [num_blocks, H_kv, block_size, d]")
    return k_pages.shape[0], k_pages.shape[2]


def pool_paged(k_full, v_full, full_off, P, T, N, gate, k_pages, v_pages, block_table, length,
               w: int, layer: int, l0: int, stream=None):
    """speechkv_pool_paged: as pool(), into pages [num_blocks, H_kv,
    block_size, d] through block_table int32 [B, max_blocks]."""
    B, max_blocks = block_table.shape
    full_rows, H_kv, d = k_full.shape
    nb, bs = _pages(k_pages, block_table)
    _check(load().speechkv_pool_paged(
        _ptr(k_full), _ptr(v_full), _ptr(full_off), _ptr(P), _ptr(T), _ptr(N), _ptr(gate),
        _ptr(k_pages), _ptr(v_pages), _ptr(block_table), max_blocks, bs, nb, _ptr(length), B,
        full_rows, H_kv, d, w, layer, l0, _dtype_code(k_full), _stream(stream)),
        "speechkv_pool_paged")


def append_paged(k_new, v_new, k_pages, v_pages, block_table, length, w: int, layer: int,
                 l0: int, stream=None):
    """speechkv_append_paged: as append(), into pages through block_table."""
    B, H_kv, d = k_new.shape
    nb, bs = _pages(k_pages, block_table)
    _check(load().speechkv_append_paged(
        _ptr(k_new), _ptr(v_new), _ptr(k_pages), _ptr(v_pages), _ptr(block_table),
        block_table.shape[1], bs, nb, _ptr(length), B, H_kv, d, w, layer, l0,
        _dtype_code(k_new), _stream(stream)),
        "speechkv_append_paged")


def decode_step_paged(q, k_new, v_new, k_pages, v_pages, block_table, length, out, workspace,
                      w: int, layer: int, l0: int, scale: float = 0.0, grid_ctas: int = 0,
                      flags: int = 0, stream=None):
    """speechkv_decode_step_paged: as decode_step(), over pages through
    block_table."""
    B, H_q, d = q.shape
    H_kv = k_new.shape[1]
    nb, bs = _pages(k_pages, block_table)
    _check(load().speechkv_decode_step_paged(
        _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_pages), _ptr(v_pages), _ptr(block_table),
        block_table.shape[1], bs, nb, _ptr(length), _ptr(out), float(scale), B, H_q, H_kv, d, w,
        layer, l0, grid_ctas, _ptr(workspace), workspace.numel() * workspace.element_size(),
        _dtype_code(q), flags, _stream(stream)),
        "speechkv_decode_step_paged")


def pool_hidden(h_full, full_off, P, T, N, gate, h_out, out_off, length, w: int, stream=None):
    """speechkv_pool_hidden: h_full [full_rows, d_model] -> h_out
    [out_rows, d_model] (HS-compression variant); full_off/out_off int64
    [B+1]; P/T/N/length int32 [B]; gate fp32 [d_model]."""
    B = length.numel()
    full_rows, d_model = h_full.shape
    _check(load().speechkv_pool_hidden(
        _ptr(h_full), _ptr(full_off), _ptr(P), _ptr(T), _ptr(N), _ptr(gate), _ptr(h_out),
        _ptr(out_off), _ptr(length), B, full_rows, h_out.shape[0], d_model, w,
        _dtype_code(h_full), _stream(stream)),
        "speechkv_pool_hidden")


def prefill_attn(q, q_off, P, T, N, k_cache, v_cache, cache_off, out, w: int, layer: int,
                 l0: int, H_kv: int, scale: float = 0.0, stream=None):
    """speechkv_prefill_attn: q/out [q_rows, H_q, d] (bf16, token-major
    prompt queries); q_off/cache_off int64 [B+1]; P/T/N int32 [B]; the
    caches as speechkv_pool wrote them (their element count fixes
    cache_rows)."""
    q_rows, H_q, d = q.shape
    B = P.numel()
    cache_rows = k_cache.numel() // (H_kv * d)
    _check(load().speechkv_prefill_attn(
        _ptr(q), _ptr(q_off), q_rows, _ptr(P), _ptr(T), _ptr(N), _ptr(k_cache), _ptr(v_cache),
        _ptr(cache_off), cache_rows, _ptr(out), float(scale), B, H_q, H_kv, d, w, layer, l0,
        _dtype_code(q), _stream(stream)),
        "speechkv_prefill_attn")


def prefill_attn_paged(q, q_off, P, T, N, k_pages, v_pages, block_table, out, w: int,
                       layer: int, l0: int, scale: float = 0.0, stream=None):
    """speechkv_prefill_attn_paged: as prefill_attn(), over pages
    [num_blocks, H_kv, block_size, d] through block_table [B, max_blocks]."""
    q_rows, H_q, d = q.shape
    B = P.numel()
    H_kv = k_pages.shape[1]
    nb, bs = _pages(k_pages, block_table)
    _check(load().speechkv_prefill_attn_paged(
        _ptr(q), _ptr(q_off), q_rows, _ptr(P), _ptr(T), _ptr(N), _ptr(k_pages), _ptr(v_pages),
        _ptr(block_table), block_table.shape[1], bs, nb, _ptr(out), float(scale), B, H_q, H_kv,
        d, w, layer, l0, _dtype_code(q), _stream(stream)),
        "speechkv_prefill_attn_paged")


def check_device_error(stream=None) -> int:
    """Synchronise the stream and return (and clear) the device error status."""
    return load().speechkv_check_device_error(_stream(stream))


def selftest_timeout(stream=None):
    """Launch the bounded-wait self-test (it records ERR_TIMEOUT after ~1 s)."""
    _check(load().speechkv_selftest_timeout(_stream(stream)), "speechkv_selftest_timeout")
