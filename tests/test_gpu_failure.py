"""The failure path every kernel shares, exercised without a fault: a bounded
wait that runs out records SPEECHKV_ERR_TIMEOUT in the device error word, the
kernel returns normally, the host reads (and clears) the status, and the
context keeps working -- a decode step right after still matches the oracle.
The wait that runs out is on an mbarrier phase that nothing completes
(speechkv_selftest_timeout); no trap, no bad address, no endless loop."""
import time

import torch
import pytest

from paper_2607_06827_gb300 import inputs
from tests import harness as H

pytestmark = pytest.mark.gpu


def test_bounded_wait_reports_timeout_and_context_survives(oracle):
    H.require_gpu()
    sk = H.lib()
    assert sk.check_device_error() == sk.OK  # a clean start
    t0 = time.time()
    sk.selftest_timeout()
    status = sk.check_device_error()
    waited = time.time() - t0
    assert status == sk.ERR_TIMEOUT, sk.status_string(status)
    assert 0.9 < waited < 60.0  # the wait limit is 1 s of the GPU's global timer
    assert sk.check_device_error() == sk.OK  # the read cleared it

    # the context is still usable: the tiny fp32 workload, one fused step
    wl = inputs.tiny_fp32()
    L, (ks, vs, gate) = H.gpu_prefill(wl, 0, extra_rows=1)
    oc = H.oracle_prefill(oracle, wl, 0, 1, ks, vs, gate)
    ws = sk.new_workspace(wl.B, wl.H_q, wl.H_kv, wl.d)
    q, kn, vn = inputs.step_qkv(wl, 0, 0)
    out = torch.empty_like(q, device="cuda")
    sk.decode_step(q.cuda(), kn.cuda(), vn.cuda(), L.k, L.v, L.cache_off, L.len, out, ws, wl.w,
                   0, wl.l0)
    assert sk.check_device_error() == sk.OK
    for b in range(wl.B):
        Kc, Vc, n = oc[b]
        n = oracle.append_request(Kc, Vc, n, H.f64(kn[b]), H.f64(vn[b]))
        ref = oracle.decode_attn_request(H.f64(q[b]), Kc[:n], Vc[:n], storage=oracle.STORE_F32)
        H.assert_close(H.f64(out[b]), ref, "f32", f"request {b} after the timeout")
