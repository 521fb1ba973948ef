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

import pytest
import torch

from paper_2607_06827_gb300 import inputs
from tests import harness as H

pytestmark = pytest.mark.gpu


def _noalloc(lib, sk, q, kn, vn, L, out, wl, layer, grid=0):
    s = torch.cuda.current_stream().cuda_stream
    return lib.speechkv_decode_step_noalloc(
        q.data_ptr(), kn.data_ptr(), vn.data_ptr(), L.k.data_ptr(), L.v.data_ptr(),
        L.cache_off.data_ptr(), L.len.data_ptr(), out.data_ptr(), 0.0, wl.B, wl.H_q, wl.H_kv,
        wl.d, wl.w, layer, wl.l0, grid, sk.BF16, 0, s)


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
