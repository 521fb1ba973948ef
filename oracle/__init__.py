"""SpeechKV CPU oracle: ctypes wrapper around ``speechkv_oracle.c``.

TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The CUDA product path never imports it, and the two share no code.

The C library is plain fp64 loops written from the paper's definitions
(Sec. III-B: Eq. (pool) and Eq. (attn)); this module only marshals numpy
arrays.  Layouts are token-major: a request's keys are ``[rows, H_kv, d]``,
queries and outputs ``[H_q, d]``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "speechkv_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

STORE_EXACT, STORE_F32, STORE_BF16 = 0, 1, 2

_D = ctypes.POINTER(ctypes.c_double)


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no GPU needed).  Returns the .so path."""
    stale = (not os.path.exists(_LIB_PATH)
             or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC))
    if force or stale:
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared",
                        "-fno-fast-math", "-o", tmp, _SRC, "-lm"], check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        # SPEECHKV_ORACLE_LIB names another build of this file's C source;
        # only the planted-mistake test sets it, to run the pins against a
        # copy of the oracle with one deliberate error.
        lib = ctypes.CDLL(os.environ.get("SPEECHKV_ORACLE_LIB") or build())
        lib.oracle_round_bf16.restype = ctypes.c_double
        lib.oracle_round_bf16.argtypes = [ctypes.c_double]
        lib.oracle_round_f32.restype = ctypes.c_double
        lib.oracle_round_f32.argtypes = [ctypes.c_double]
        lib.oracle_effective_window.restype = ctypes.c_int32
        lib.oracle_effective_window.argtypes = [ctypes.c_int32] * 3
        lib.oracle_compressed_len.restype = ctypes.c_int64
        lib.oracle_compressed_len.argtypes = [ctypes.c_int32] * 7
        lib.oracle_pool_request.restype = ctypes.c_int64
        lib.oracle_pool_request.argtypes = [
            _D, _D, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
            ctypes.c_int32, ctypes.c_int32, _D, ctypes.c_int32,
            ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, _D, _D, _D]
        lib.oracle_append_request.restype = ctypes.c_int64
        lib.oracle_append_request.argtypes = [
            _D, _D, ctypes.c_int64, ctypes.c_int64, _D, _D,
            ctypes.c_int32, ctypes.c_int32]
        lib.oracle_decode_attn_request.restype = ctypes.c_int32
        lib.oracle_decode_attn_request.argtypes = [
            _D, _D, _D, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
            ctypes.c_int32, ctypes.c_double, ctypes.c_int32, _D, _D]
        lib.oracle_prefill_position.restype = ctypes.c_int64
        lib.oracle_prefill_position.argtypes = [ctypes.c_int32] * 4 + [ctypes.c_int64]
        lib.oracle_prefill_attn_request.restype = ctypes.c_int32
        lib.oracle_prefill_attn_request.argtypes = [
            _D, _D, _D, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
            ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
            ctypes.c_double, ctypes.c_int32, _D]
        _lib = lib
        return lib


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(_D)


def round_bf16(x: float) -> float:
    return _load().oracle_round_bf16(float(x))


def round_f32(x: float) -> float:
    return _load().oracle_round_f32(float(x))


def effective_window(w: int, layer: int, l0: int) -> int:
    return _load().oracle_effective_window(w, layer, l0)


def compressed_len(P: int, T: int, N: int, G: int, w: int, layer: int,
                   l0: int) -> int:
    return _load().oracle_compressed_len(P, T, N, G, w, layer, l0)


def pool_request(K, V, P: int, T: int, N: int, gate, w: int, layer: int,
                 l0: int, storage: int = STORE_EXACT, want_alpha: bool = False):
    """Eq. (pool) on one request.  K, V: [P+T+N, H_kv, d]; gate: [H_kv, d].

    Returns (K_out, V_out) of shape [P + n + N, H_kv, d] (and alpha [T, H_kv]
    when ``want_alpha``)."""
    K, V, gate = _f64(K), _f64(V), _f64(gate)
    S, H_kv, d = K.shape
    assert S == P + T + N and V.shape == K.shape and gate.shape == (H_kv, d)
    rows = compressed_len(P, T, N, 0, w, layer, l0)
    Ko = np.zeros((max(rows, 0), H_kv, d))
    Vo = np.zeros_like(Ko)
    alpha = np.zeros((T, H_kv)) if want_alpha else None
    got = _load().oracle_pool_request(
        _ptr(K), _ptr(V), P, T, N, H_kv, d, _ptr(gate), w, layer, l0,
        storage, _ptr(Ko), _ptr(Vo), _ptr(alpha))
    if got != rows:
        raise ValueError(f"oracle_pool_request failed ({got})")
    return (Ko, Vo, alpha) if want_alpha else (Ko, Vo)


def append_request(K_cache, V_cache, n: int, k_new, v_new) -> int:
    """Append one token's [H_kv, d] key/value as row ``n`` (arrays edited in
    place).  Returns the new row count, or -1 when the cache is full."""
    assert K_cache.dtype == np.float64 and K_cache.flags.c_contiguous
    assert V_cache.dtype == np.float64 and V_cache.flags.c_contiguous
    cap, H_kv, d = K_cache.shape
    k_new, v_new = _f64(k_new), _f64(v_new)
    return _load().oracle_append_request(
        _ptr(K_cache), _ptr(V_cache), n, cap, _ptr(k_new), _ptr(v_new),
        H_kv, d)


def decode_attn_request(q, K, V, scale: float = 0.0,
                        storage: int = STORE_EXACT, want_probs: bool = False):
    """Eq. (attn) for one decode query.  q: [H_q, d]; K, V: [n, H_kv, d].

    Returns out [H_q, d] (and the softmax weights [H_q, n] when
    ``want_probs``)."""
    q, K, V = _f64(q), _f64(K), _f64(V)
    H_q, d = q.shape
    n, H_kv, d2 = K.shape
    assert d2 == d and V.shape == K.shape
    out = np.zeros((H_q, d))
    probs = np.zeros((H_q, n)) if want_probs else None
    rc = _load().oracle_decode_attn_request(
        _ptr(q), _ptr(K), _ptr(V), n, H_q, H_kv, d, float(scale), storage,
        _ptr(out), _ptr(probs))
    if rc != 0:
        raise ValueError("oracle_decode_attn_request: bad arguments")
    return (out, probs) if want_probs else out


def prefill_position(P: int, T: int, N: int, w_eff: int, t: int) -> int:
    """Compressed row holding prompt position t (the query's place in the
    compressed sequence for the prefill mask)."""
    r = _load().oracle_prefill_position(P, T, N, w_eff, t)
    if r < 0:
        raise ValueError("oracle_prefill_position: bad arguments")
    return r


def prefill_attn_request(Q, K, V, P: int, T: int, N: int, w_eff: int,
                         scale: float = 0.0, storage: int = STORE_EXACT):
    """Eq. (attn) at prefill with the adjusted causal mask, one request.
    Q: [P + T + N, H_q, d]; K, V: compressed [c, H_kv, d].  Returns
    out [P + T + N, H_q, d]."""
    Q, K, V = _f64(Q), _f64(K), _f64(V)
    S, H_q, d = Q.shape
    c, H_kv, d2 = K.shape
    assert S == P + T + N and d2 == d and V.shape == K.shape
    assert c == compressed_len(P, T, N, 0, w_eff, 0, 0)
    out = np.zeros((S, H_q, d))
    rc = _load().oracle_prefill_attn_request(
        _ptr(Q), _ptr(K), _ptr(V), P, T, N, w_eff, H_q, H_kv, d, float(scale),
        storage, _ptr(out))
    if rc != 0:
        raise ValueError("oracle_prefill_attn_request: bad arguments")
    return out
