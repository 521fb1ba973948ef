"""The C-ABI library builds for sm_103a, loads, and exports every entry point
include/speechkv.h declares; host-only helpers and host-side argument checks
work without a GPU (no kernel is launched here)."""
import ctypes
import os
import re

import pytest

from paper_2607_06827_gb300 import inputs
from tests import harness as H

HEADER = os.path.join(H.ROOT, "include", "speechkv.h")


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(speechkv_[a-z_]+)\s*\(", src)))


def test_header_declares_the_path():
    names = _declared()
    for n in ("speechkv_pool", "speechkv_append", "speechkv_decode_attn", "speechkv_decode_step",
              "speechkv_compressed_len", "speechkv_decode_workspace_size",
              "speechkv_check_device_error", "speechkv_status_string", "speechkv_prefill_attn"):
        assert n in names


def test_library_exports_every_declared_symbol():
    sk = H.lib()
    lib = sk.load()
    for name in _declared():
        assert hasattr(lib, name), name
        assert name in sk.SIGNATURES, f"binding lacks {name}"
    assert set(sk.SIGNATURES) == set(_declared())


_C_TO_CTYPES = {
    "int32_t": ctypes.c_int32, "int64_t": ctypes.c_int64, "uint32_t": ctypes.c_uint32,
    "size_t": ctypes.c_size_t, "float": ctypes.c_float, "speechkv_status": ctypes.c_int,
    "speechkv_dtype": ctypes.c_int, "cudaStream_t": ctypes.c_void_p,
}


def _ctype_of(decl: str):
    """ctypes class of a C parameter or return type from the header."""
    decl = " ".join(decl.replace("const ", "").split())
    if "*" in decl:
        return ctypes.c_char_p if decl.startswith("char") else ctypes.c_void_p
    base = decl.split()[0]
    return _C_TO_CTYPES[base]


def _prototypes():
    src = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    protos = {}
    for m in re.finditer(r"([A-Za-z_][\w \t\*]*?)\b(speechkv_[a-z_]+)\s*\(([^)]*)\)\s*;", src):
        params = [a.strip() for a in m.group(3).split(",") if a.strip() and a.strip() != "void"]
        # drop the parameter name (the last identifier), keep the type
        types = [re.sub(r"\b\w+$", "", a).strip() for a in params]
        protos[m.group(2)] = (m.group(1).strip(), types)
    return protos


def test_binding_signatures_match_header():
    """Every ctypes signature of the binding has the header's argument count
    and, position by position, the same kind of value (pointer, 32- or
    64-bit integer, size_t, float, enum); a mismatch would pass wrong values
    across the boundary without any error."""
    sk = H.lib()
    protos = _prototypes()
    assert set(protos) == set(sk.SIGNATURES)
    for name, (ret, types) in protos.items():
        restype, argtypes = sk.SIGNATURES[name]
        assert restype is _ctype_of(ret), f"{name}: return {ret}"
        assert len(argtypes) == len(types), f"{name}: {len(argtypes)} args bound, {len(types)} declared"
        for i, (got, decl) in enumerate(zip(argtypes, types)):
            assert got is _ctype_of(decl), f"{name}: argument {i} ({decl}) bound as {got.__name__}"


def test_compressed_len_matches_oracle(oracle):
    sk = H.lib()
    for wl in (inputs.qwen_ragged(), inputs.tiny_fp32(), inputs.qwen_single(),
               inputs.qwen_long_audio(20, 8)):
        for layer in (0, wl.l0 - 1 if wl.l0 > 0 else 0, wl.l0, wl.L - 1):
            for b in range(wl.B):
                args = (wl.P[b], wl.T[b], wl.N[b], wl.G[b], wl.w, layer, wl.l0)
                assert sk.compressed_len(*args) == oracle.compressed_len(*args)
    for T in range(0, 50):
        for w in range(1, 9):
            assert sk.compressed_len(3, T, 2, 1, w, 1, 1) == oracle.compressed_len(3, T, 2, 1, w, 1, 1)
    assert sk.compressed_len(0, 3, 0, 0, 0, 0, 0) == -1
    assert sk.compressed_len(0, -3, 0, 0, 4, 0, 0) == -1


def test_status_strings():
    sk = H.lib()
    assert sk.status_string(sk.OK) == "ok"
    assert "capacity" in sk.status_string(sk.ERR_CAPACITY)
    assert sk.status_string(99) == "unknown status"


def test_host_argument_checks_without_gpu():
    sk = H.lib()
    lib = sk.load()
    z = None
    # decode: bad window, bad head split, unsupported head dim, B = 0 no-op
    args = lambda B, H_q, H_kv, d, w: (z, z, z, z, z, z, 0.0, B, H_q, H_kv, d, w, 0, 0, 0, z, 0,  # noqa: E731
                                       sk.BF16, 0, z)
    assert lib.speechkv_decode_attn(*args(1, 8, 4, 128, 0)) == sk.ERR_INVALID_ARG
    assert lib.speechkv_decode_attn(*args(1, 7, 4, 128, 4)) == sk.ERR_INVALID_ARG
    assert lib.speechkv_decode_attn(*args(1, 8, 4, 96, 4)) == sk.ERR_UNSUPPORTED
    assert lib.speechkv_decode_attn(*args(0, 8, 4, 128, 4)) == sk.OK
    assert lib.speechkv_decode_attn(*args(1, 8, 4, 128, 4)) == sk.ERR_INVALID_ARG  # NULLs
    step = lambda B, fl: (z,) * 8 + (0.0, B, 8, 4, 128, 4, 0, 0, 0, z, 0, sk.BF16, fl, z)  # noqa: E731
    assert lib.speechkv_decode_step(*step(0, 0)) == sk.OK
    assert lib.speechkv_decode_step(*step(1, 0)) == sk.ERR_INVALID_ARG          # NULLs
    assert lib.speechkv_decode_step(*step(1, 4)) == sk.ERR_INVALID_ARG          # bad flag
    # append / pool
    assert lib.speechkv_append(z, z, z, z, z, z, 1, 8, 128, 4, -1, 0, sk.BF16, z) == sk.ERR_INVALID_ARG
    assert lib.speechkv_append(z, z, z, z, z, z, 0, 8, 128, 4, 0, 0, sk.BF16, z) == sk.OK
    assert lib.speechkv_pool(*([z] * 11), 1, 10, 8, 128, 0, 0, 0, sk.BF16, z) == sk.ERR_INVALID_ARG
    assert lib.speechkv_pool(*([z] * 11), 1, 10, 8, 80, 4, 0, 0, sk.BF16, z) == sk.ERR_UNSUPPORTED
    assert lib.speechkv_pool(*([z] * 11), 0, 0, 8, 128, 4, 0, 0, sk.BF16, z) == sk.OK
    # hidden-state pooling: d_model * element size a multiple of 16 bytes, <= 16 KB
    ph = lambda B, d_model, w, dt: (*([z] * 9), B, 10, 10, d_model, w, dt, z)  # noqa: E731
    assert lib.speechkv_pool_hidden(*ph(1, 2048, 0, sk.BF16)) == sk.ERR_INVALID_ARG
    assert lib.speechkv_pool_hidden(*ph(1, 2044, 4, sk.BF16)) == sk.ERR_UNSUPPORTED
    assert lib.speechkv_pool_hidden(*ph(1, 16384, 4, sk.BF16)) == sk.ERR_UNSUPPORTED
    assert lib.speechkv_pool_hidden(*ph(0, 2048, 4, sk.BF16)) == sk.OK
    assert lib.speechkv_pool_hidden(*ph(1, 2048, 4, sk.BF16)) == sk.ERR_INVALID_ARG  # NULLs
    assert lib.speechkv_pool_hidden(*ph(1, 4096, 4, sk.F32)) == sk.ERR_INVALID_ARG   # NULLs
    # paged caches: block size a power of two, table and page count required
    pp = lambda B, mb, bs, nb: (*([z] * 9), z, mb, bs, nb, z, B, 10, 8, 128, 4, 0, 0, sk.BF16, z)  # noqa: E731
    assert lib.speechkv_pool_paged(*pp(0, 4, 64, 8)) == sk.OK
    assert lib.speechkv_pool_paged(*pp(1, 4, 64, 8)) == sk.ERR_INVALID_ARG        # no table
    ap = lambda B, bs: (z, z, z, z, z, 4, bs, 8, z, B, 8, 128, 4, 0, 0, sk.BF16, z)  # noqa: E731
    assert lib.speechkv_append_paged(*ap(0, 64)) == sk.OK
    assert lib.speechkv_append_paged(*ap(1, 64)) == sk.ERR_INVALID_ARG
    dp = lambda B: (*([z] * 6), 4, 48, 8, z, z, 0.0, B, 16, 8, 128, 4, 0, 0, 0, z, 0, sk.BF16, 0, z)  # noqa: E731
    assert lib.speechkv_decode_step_paged(*dp(0)) == sk.OK
    assert lib.speechkv_decode_step_paged(*dp(1)) == sk.ERR_INVALID_ARG          # no table
    # prefill attention: bf16 and d = 64 or 128 only; 32-bit tensor-copy coordinates
    pf = lambda B, q_rows, cache_rows, H_q, H_kv, d, w, dt: (  # noqa: E731
        z, z, q_rows, z, z, z, z, z, z, cache_rows, z, 0.0, B, H_q, H_kv, d, w, 0, 0, dt, z)
    assert lib.speechkv_prefill_attn(*pf(1, 10, 10, 16, 8, 128, 4, sk.F32)) == sk.ERR_UNSUPPORTED
    assert lib.speechkv_prefill_attn(*pf(1, 10, 10, 16, 8, 96, 4, sk.BF16)) == sk.ERR_UNSUPPORTED
    assert lib.speechkv_prefill_attn(*pf(1, 10, 10, 16, 8, 128, 0, sk.BF16)) == sk.ERR_INVALID_ARG
    assert lib.speechkv_prefill_attn(*pf(1, 10, 10, 12, 8, 128, 4, sk.BF16)) == sk.ERR_INVALID_ARG
    assert lib.speechkv_prefill_attn(*pf(sk.MAX_BATCH + 1, 10, 10, 16, 8, 128, 4, sk.BF16)) == sk.ERR_INVALID_ARG
    assert lib.speechkv_prefill_attn(*pf(1, 1 << 31, 10, 16, 8, 128, 4, sk.BF16)) == sk.ERR_UNSUPPORTED
    assert lib.speechkv_prefill_attn(*pf(1, 10, 1 << 28, 16, 8, 128, 4, sk.BF16)) == sk.ERR_UNSUPPORTED
    assert lib.speechkv_prefill_attn(*pf(0, 10, 10, 16, 8, 128, 4, sk.BF16)) == sk.OK
    assert lib.speechkv_prefill_attn(*pf(1, 10, 10, 16, 8, 128, 4, sk.BF16)) == sk.ERR_INVALID_ARG  # NULLs
    assert lib.speechkv_prefill_attn(*pf(1, 10, 10, 16, 8, 64, 4, sk.BF16)) == sk.ERR_INVALID_ARG  # NULLs
    # paged prefill: pages of at least 8 rows; table required
    fake = ctypes.c_void_p(256)  # never dereferenced: every call below fails a host check
    pfp = lambda B, tab, bs, d: (  # noqa: E731
        z, z, 10, z, z, z, z, z, tab, 4, bs, 8, z, 0.0, B, 16, 8, d, 4, 0, 0, sk.BF16, z)
    assert lib.speechkv_prefill_attn_paged(*pfp(0, z, 16, 128)) == sk.OK
    assert lib.speechkv_prefill_attn_paged(*pfp(1, z, 16, 128)) == sk.ERR_INVALID_ARG   # no table
    assert lib.speechkv_prefill_attn_paged(*pfp(1, fake, 4, 128)) == sk.ERR_UNSUPPORTED  # 4-row pages
    assert lib.speechkv_prefill_attn_paged(*pfp(1, fake, 16, 96)) == sk.ERR_UNSUPPORTED
    assert lib.speechkv_prefill_attn_paged(*pfp(1, fake, 16, 128)) == sk.ERR_INVALID_ARG  # NULLs


def test_workspace_size_explicit_grid():
    sk = H.lib()
    lib = sk.load()
    B, H_q, H_kv, d, grid = 8, 16, 8, 128, 152
    n = lib.speechkv_decode_workspace_size(B, H_q, H_kv, d, grid)
    slot = 2 * 128 + 2 * 2                        # o [G][d], m [G], l [G]
    counters = -(-(B * H_kv + 1) * 4 // 256) * 256  # per (request, head) + 1
    assert n == counters + (grid + B * H_kv) * slot * 4
    assert lib.speechkv_decode_workspace_size(B, 7, H_kv, d, grid) == 0
    assert lib.speechkv_decode_workspace_size(B, H_q, H_kv, 100, grid) == 0
