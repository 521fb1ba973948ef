"""The allocation-free decode step, checked against the regular one.

speechkv_decode_step_noalloc serves callers that may not allocate device
memory -- a plug-in whose host process's memory pool owns the whole GPU, or a
path that must never enter an allocator -- by keeping its split-K scratch in a
fixed array the library owns.  These tests call it through the C ABI and
compare two decode steps in a row with speechkv_decode_step (which takes a
caller-owned workspace) on identical inputs.

This file is collected last on purpose: if it fails, a run that stops at the
first failure has already run every other test.
"""

import numpy as np
import pytest
import torch

from paper_2607_06827_gb300 import inputs
from tests import harness as H

pytestmark = pytest.mark.gpu


def _noalloc(lib, sk, q, kn, vn, L, out, wl, layer, grid=0, flags=0):
    s = torch.cuda.current_stream().cuda_stream
    return lib.speechkv_decode_step_noalloc(
        q.data_ptr(), kn.data_ptr(), vn.data_ptr(), L.k.data_ptr(), L.v.data_ptr(),
        L.cache_off.data_ptr(), L.len.data_ptr(), out.data_ptr(), 0.0, wl.B, wl.H_q, wl.H_kv,
        wl.d, wl.w, layer, wl.l0, grid, sk.BF16, flags, s)


@pytest.mark.parametrize("grid", [0, 7])
def test_noalloc_matches_decode_step_two_calls(grid):
    H.require_gpu()
    sk = H.lib()
    lib = sk.load()
    wl = inputs.qwen_ragged(B=6)
    layer = wl.l0
    ref, _ = H.gpu_prefill(wl, layer, extra_rows=2)   # regular entry point
    nal, _ = H.gpu_prefill(wl, layer, extra_rows=2)   # allocation-free one
    ws = sk.new_workspace(wl.B, wl.H_q, wl.H_kv, wl.d, grid)
    for step in range(2):                             # two calls in a row
        q, kn, vn = (x.cuda() for x in inputs.step_qkv(wl, layer, step))
        out_ref, out_nal = torch.empty_like(q), torch.empty_like(q)
        sk.decode_step(q, kn, vn, ref.k, ref.v, ref.cache_off, ref.len, out_ref, ws, wl.w,
                       layer, wl.l0, grid_ctas=grid)
        assert _noalloc(lib, sk, q, kn, vn, nal, out_nal, wl, layer, grid) == sk.OK
        torch.cuda.synchronize()
        assert torch.equal(nal.len, ref.len)
        assert torch.equal(nal.k, ref.k) and torch.equal(nal.v, ref.v)
        H.assert_close(H.f64(out_nal), H.f64(out_ref), "bf16", f"call {step}")
    assert sk.check_device_error() == sk.OK


def test_noalloc_refuses_batches_beyond_its_scratch():
    H.require_gpu()
    sk = H.lib()
    lib = sk.load()
    t = torch.zeros(64, dtype=torch.bfloat16, device="cuda")
    off = torch.zeros(8, dtype=torch.int64, device="cuda")
    ln = torch.zeros(8, dtype=torch.int32, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    p = t.data_ptr()
    # 512 requests x 16 KV heads with groups of 4: several times the scratch
    status = lib.speechkv_decode_step_noalloc(p, p, p, p, p, off.data_ptr(), ln.data_ptr(), p,
                                              0.0, 512, 64, 16, 128, 4, 8, 8, 0, sk.BF16, 0, s)
    assert status == sk.ERR_WORKSPACE
    torch.cuda.synchronize()
    assert sk.check_device_error() == sk.OK


def test_noalloc_matches_oracle_with_overlap_flag(oracle):
    """Two allocation-free steps in a row with SPEECHKV_OVERLAP_PRIOR, each
    against the oracle's pooling -> append -> attention (Eq. (pool),
    Eq. (attn)); the flag is accepted and changes nothing in the results."""
    H.require_gpu()
    sk = H.lib()
    lib = sk.load()
    wl = inputs.qwen_ragged(B=4)
    layer = wl.l0
    L, (ks, vs, gate) = H.gpu_prefill(wl, layer, extra_rows=2)
    oc = H.oracle_prefill(oracle, wl, layer, 2, ks, vs, gate)
    for step in range(2):
        q, kn, vn = inputs.step_qkv(wl, layer, step)
        out = torch.empty_like(q, device="cuda")
        assert _noalloc(lib, sk, q.cuda(), kn.cuda(), vn.cuda(), L, out, wl, layer,
                        flags=sk.OVERLAP_PRIOR) == sk.OK
        torch.cuda.synchronize()
        ref = []
        for b in range(wl.B):
            Kc, Vc, n = oc[b]
            n = oracle.append_request(Kc, Vc, n, H.f64(kn[b]), H.f64(vn[b]))
            oc[b][2] = n
            assert int(L.len[b]) == n
            ref.append(oracle.decode_attn_request(H.f64(q[b]), Kc[:n], Vc[:n],
                                                  storage=oracle.STORE_BF16))
        H.assert_close(H.f64(out), np.stack(ref), "bf16", f"call {step}")
    assert sk.check_device_error() == sk.OK


def test_noalloc_after_a_reported_device_error():
    """A call on a full cache reports SPEECHKV_ERR_CAPACITY on the device;
    once that status has been read, the next allocation-free call matches
    the regular step again."""
    H.require_gpu()
    sk = H.lib()
    lib = sk.load()
    wl = inputs.qwen_ragged(B=3)
    layer = wl.l0
    full, _ = H.gpu_prefill(wl, layer, extra_rows=0)   # capacity == rows: full
    q, kn, vn = (x.cuda() for x in inputs.step_qkv(wl, layer, 0))
    out = torch.empty_like(q)
    assert _noalloc(lib, sk, q, kn, vn, full, out, wl, layer) == sk.OK
    assert sk.check_device_error() == sk.ERR_CAPACITY
    ref, _ = H.gpu_prefill(wl, layer, extra_rows=1)
    nal, _ = H.gpu_prefill(wl, layer, extra_rows=1)
    ws = sk.new_workspace(wl.B, wl.H_q, wl.H_kv, wl.d)
    out_ref, out_nal = torch.empty_like(q), torch.empty_like(q)
    sk.decode_step(q, kn, vn, ref.k, ref.v, ref.cache_off, ref.len, out_ref, ws, wl.w, layer,
                   wl.l0)
    assert _noalloc(lib, sk, q, kn, vn, nal, out_nal, wl, layer) == sk.OK
    torch.cuda.synchronize()
    assert torch.equal(nal.len, ref.len)
    H.assert_close(H.f64(out_nal), H.f64(out_ref), "bf16", "after the error")
    assert sk.check_device_error() == sk.OK


def test_noalloc_argument_errors():
    """Argument errors found by the host checks (a bad window, a negative
    l0) are returned as a status, and nothing reaches the device error
    word."""
    H.require_gpu()
    sk = H.lib()
    lib = sk.load()
    t = torch.zeros(4096, dtype=torch.bfloat16, device="cuda")
    off = torch.zeros(2, dtype=torch.int64, device="cuda")
    ln = torch.zeros(1, dtype=torch.int32, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    p = t.data_ptr()
    for w, l0 in ((0, 8), (4, -1)):
        status = lib.speechkv_decode_step_noalloc(p, p, p, p, p, off.data_ptr(), ln.data_ptr(),
                                                  p, 0.0, 1, 16, 8, 128, w, 8, l0, 0, sk.BF16,
                                                  0, s)
        assert status == sk.ERR_INVALID_ARG
    assert sk.check_device_error() == sk.OK
