"""GPU parity of speechkv_pool_hidden -- the HS-compression variant
(Sec. IV-A): Eq. (pool)'s window softmax pooling applied once to whole
hidden vectors -- against the oracle's pooling with a single head of width
d_model and the hidden states as both keys and values.  Text rows and w = 1
are bit-exact; pooled rows within the storage tolerances."""
import numpy as np
import pytest
import torch

from paper_2607_06827_gb300 import inputs
from tests import harness as H

pytestmark = pytest.mark.gpu


def _wl(dtype="bf16", P=(0, 16, 5), T=(375, 130, 0), N=(32, 7, 40), w=4, seed=3001):
    return inputs.Workload(name="hs", dtype=dtype, L=28, l0=8, w=w, H_q=16, H_kv=8, d=128,
                           P=list(P), T=list(T), N=list(N), G=[0] * len(T), steps=0, seed=seed)


def _off(rows):
    off = np.zeros(len(rows) + 1, dtype=np.int64)
    off[1:] = np.cumsum(rows)
    return off


def _run(wl, d_model, slack=0, gate_scale=1.0):
    H.require_gpu()
    sk = H.lib()
    hs = [inputs.hidden_states(wl, b, d_model) for b in range(wl.B)]
    gate = inputs.hidden_gate(wl, d_model, gate_scale)
    rows = [sk.compressed_len(p, t, n, 0, wl.w, 0, 0) + slack for p, t, n in zip(wl.P, wl.T, wl.N)]
    full_off, out_off = _off(wl.full_rows()), _off(rows)
    h = torch.cat(hs).cuda()
    out = torch.full((int(out_off[-1]), d_model), 5.0, dtype=h.dtype, device="cuda")
    ln = torch.zeros(wl.B, dtype=torch.int32, device="cuda")
    P, T, N = H.lengths_dev(wl)
    sk.pool_hidden(h, torch.from_numpy(full_off).cuda(), P, T, N, torch.from_numpy(gate).cuda(),
                   out, torch.from_numpy(out_off).cuda(), ln, wl.w)
    return sk, hs, gate, out, out_off, ln


def _check(oracle, wl, d_model, hs, gate, out, out_off, ln):
    store = oracle.STORE_F32 if wl.dtype == "f32" else oracle.STORE_BF16
    for b in range(wl.B):
        hb = H.f64(hs[b])[:, None, :]
        Ko, Vo = oracle.pool_request(hb, hb, wl.P[b], wl.T[b], wl.N[b], gate[None, :].astype(np.float64),
                                     wl.w, 0, 0, storage=store)
        n = Ko.shape[0]
        assert int(ln[b]) == n
        got = H.f64(out[out_off[b]:out_off[b] + n])
        H.assert_close(got, Ko[:, 0, :], wl.dtype, f"request {b}")
        # text rows (and everything at w = 1) are copies of the input rows
        p, t, nn = wl.P[b], wl.T[b], wl.N[b]
        npool = n - p - nn
        src = H.f64(hs[b])
        assert np.array_equal(got[:p], src[:p])
        assert np.array_equal(got[p + npool:], src[p + t:])
        if wl.w == 1:
            assert np.array_equal(got, src)


@pytest.mark.parametrize("w", [4, 8, 3, 1])
def test_hs_pool_bf16_qwen_width(oracle, w):
    """Qwen3-1.7B hidden size (2048), bf16, ragged requests (speech only,
    a text prefix, text only)."""
    wl = _wl(w=w)
    sk, hs, gate, out, out_off, ln = _run(wl, 2048)
    assert sk.check_device_error() == sk.OK
    _check(oracle, wl, 2048, hs, gate, out, out_off, ln)


@pytest.mark.parametrize("d_model", [512, 768, 4096])
def test_hs_pool_fp32(oracle, d_model):
    """fp32 storage (tolerance 1e-5), two and four vectors per lane (768:
    a team of three warps rounded up to four)."""
    wl = _wl(dtype="f32", P=(3, 0), T=(77, 9), N=(2, 5), w=4, seed=3002)
    sk, hs, gate, out, out_off, ln = _run(wl, d_model)
    assert sk.check_device_error() == sk.OK
    _check(oracle, wl, d_model, hs, gate, out, out_off, ln)


@pytest.mark.parametrize("d_model,w", [(256, 4), (512, 3), (1024, 4), (1536, 4), (2560, 3),
                                       (4096, 4), (5120, 4), (8192, 5)])
def test_hs_pool_bf16_row_widths(oracle, d_model, w):
    """Rows of 0.5 to 16 KB (one to four vectors per lane, teams of one to
    eight warps), including widths whose team is rounded up to the next
    compiled size (1536: 3 -> 4 warps; 2560: 3 -> 4; 5120: 5 -> 8); w = 5
    splits every window into a full group of frames and a ragged one."""
    wl = _wl(P=(2, 0), T=(151, 64), N=(3, 9), w=w, seed=3005)
    sk, hs, gate, out, out_off, ln = _run(wl, d_model)
    assert sk.check_device_error() == sk.OK
    _check(oracle, wl, d_model, hs, gate, out, out_off, ln)


def test_hs_pool_long_requests(oracle):
    """Requests long enough that every CTA pools many rows (the staging
    ring of each CTA is reused many times over)."""
    wl = _wl(P=(0, 9), T=(30000, 7001), N=(64, 3), w=4, seed=3006)
    sk, hs, gate, out, out_off, ln = _run(wl, 2048)
    assert sk.check_device_error() == sk.OK
    _check(oracle, wl, 2048, hs, gate, out, out_off, ln)


def test_hs_pool_peaked_gate(oracle):
    """A gate sixteen times larger: near-one-hot weights in every window."""
    wl = _wl(w=4, seed=3003)
    sk, hs, gate, out, out_off, ln = _run(wl, 2048, gate_scale=16.0)
    assert sk.check_device_error() == sk.OK
    _check(oracle, wl, 2048, hs, gate, out, out_off, ln)


def test_hs_pool_leaves_slack_rows_and_reports_capacity():
    """Rows past a request's pooled rows keep their contents; a request
    whose capacity is too small is clamped and reported."""
    wl = _wl(w=4, seed=3004)
    sk, hs, gate, out, out_off, ln = _run(wl, 2048, slack=3)
    assert sk.check_device_error() == sk.OK
    for b in range(wl.B):
        n = int(ln[b])
        assert torch.all(out[out_off[b] + n:out_off[b + 1]] == 5.0)
    # capacity one row short for every request
    H.require_gpu()
    rows = [sk.compressed_len(p, t, n, 0, wl.w, 0, 0) - 1 for p, t, n in zip(wl.P, wl.T, wl.N)]
    out_off2 = _off(rows)
    h = torch.cat(hs).cuda()
    out2 = torch.zeros((int(out_off2[-1]), 2048), dtype=h.dtype, device="cuda")
    ln2 = torch.zeros(wl.B, dtype=torch.int32, device="cuda")
    P, T, N = H.lengths_dev(wl)
    sk.pool_hidden(h, torch.from_numpy(_off(wl.full_rows())).cuda(), P, T, N,
                   torch.from_numpy(gate).cuda(), out2, torch.from_numpy(out_off2).cuda(), ln2, wl.w)
    assert sk.check_device_error() == sk.ERR_CAPACITY
    assert ln2.cpu().tolist() == rows
