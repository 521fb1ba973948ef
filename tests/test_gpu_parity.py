"""GPU parity: libspeechkv's kernels against the CPU oracle, element by
element, on the same seeded inputs (paper Sec. III-B, Eq. (pool) and
Eq. (attn); Sec. III-C for the prefill-once / append-per-step cache).

Tolerances: fp32 max-abs 1e-5; bf16 max-abs 2e-2 and mean-abs 2e-3 on
unit-variance inputs; lengths, offsets and copied rows bit-exact.
"""
import dataclasses
import math

import numpy as np
import pytest
import torch

from paper_2607_06827_gb300 import inputs
from tests import harness as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sk():
    H.require_gpu()
    return H.lib()


def _wl(dtype="bf16", P=(0,), T=(37,), N=(5,), G=None, w=4, l0=0, H_q=4, H_kv=2, d=64,
        seed=7, name="case"):
    G = G if G is not None else (0,) * len(T)
    return inputs.Workload(name, dtype, L=1, l0=l0, w=w, H_q=H_q, H_kv=H_kv, d=d, P=list(P),
                           T=list(T), N=list(N), G=list(G), steps=4, seed=seed)


def _ws(sk, wl, grid=0):
    return sk.new_workspace(wl.B, wl.H_q, wl.H_kv, wl.d, grid)


def _decode(sk, wl, L, q, layer, grid=0, ws=None, scale=0.0):
    out = torch.empty_like(q)
    ws = ws if ws is not None else _ws(sk, wl, grid)
    sk.decode_attn(q, L.k, L.v, L.cache_off, L.len, out, ws, wl.w, layer, wl.l0, wl.H_kv,
                   scale=scale, grid_ctas=grid)
    return out


def _oracle_attn_on_gpu_cache(oracle, wl, L, q, scale=0.0):
    """Oracle attention over the GPU's own cache rows (isolates the kernel)."""
    store = oracle.STORE_F32 if wl.dtype == "f32" else oracle.STORE_BF16
    qn = H.f64(q)
    res = []
    for b in range(wl.B):
        K, V = L.request_rows(b)
        res.append(oracle.decode_attn_request(qn[b], K, V, scale=scale, storage=store))
    return np.stack(res)


# --------------------------------------------------------------------------
# pool
# --------------------------------------------------------------------------
POOL_CASES = [
    # dtype, d, H_kv, P, T, N, w
    ("f32", 64, 2, (16,), (64,), (0,), 4),            # tiny workload shapes
    ("bf16", 128, 8, (0,), (375,), (32,), 4),         # 30 s audio, 94 entries
    ("bf16", 128, 8, (0, 3, 0), (375, 10, 0), (32, 1, 4), 4),  # ragged, T=0
    ("bf16", 128, 8, (2,), (13,), (3,), 3),           # T mod w != 0
    ("bf16", 128, 8, (1,), (3,), (2,), 4),            # T < w
    ("bf16", 64, 4, (0, 5), (40, 41), (8, 0), 8),
    ("f32", 128, 2, (0,), (50,), (6,), 2),
    ("bf16", 128, 8, (0,), (17,), (2,), 1),           # w = 1: bit-exact copy
    ("bf16", 128, 3, (0, 2), (90, 37), (5, 0), 4),    # odd H_kv: a half-empty warp chunk
    ("f32", 64, 1, (1,), (20,), (2,), 3),             # one KV head
]


@pytest.mark.parametrize("dtype,d,H_kv,P,T,N,w", POOL_CASES)
def test_pool_matches_oracle(sk, oracle, dtype, d, H_kv, P, T, N, w):
    wl = _wl(dtype, P, T, N, w=w, H_q=2 * H_kv, H_kv=H_kv, d=d)
    layer = 0
    L, (ks, vs, gate) = H.gpu_prefill(wl, layer, extra_rows=3)
    lens = L.len.cpu().numpy()
    for b in range(wl.B):
        want_len = oracle.compressed_len(P[b], T[b], N[b], 0, w, layer, wl.l0)
        assert lens[b] == want_len                          # bit-exact bookkeeping
        Ko, Vo = oracle.pool_request(H.f64(ks[b]), H.f64(vs[b]), P[b], T[b], N[b],
                                     H.f64(gate), w, layer, wl.l0)
        K, V = L.request_rows(b)
        H.assert_close(K, Ko, dtype, f"pooled K, request {b}")
        H.assert_close(V, Vo, dtype, f"pooled V, request {b}")
        # text rows (and every row when w = 1) are copied bit-exactly
        n = want_len - P[b] - N[b]
        src = H.f64(ks[b])
        np.testing.assert_array_equal(K[:P[b]], src[:P[b]])
        np.testing.assert_array_equal(K[P[b] + n:], src[P[b] + T[b]:])
        if w == 1:
            np.testing.assert_array_equal(K, src)
            np.testing.assert_array_equal(V, H.f64(vs[b]))


def test_pool_before_l0_is_bit_exact_copy(sk):
    wl = _wl("bf16", (3,), (50,), (4,), w=4, l0=5, H_q=16, H_kv=8, d=128)
    L, (ks, vs, _) = H.gpu_prefill(wl, layer=4, extra_rows=0)
    assert int(L.len[0]) == 57
    K, V = L.request_rows(0)
    np.testing.assert_array_equal(K, H.f64(ks[0]))
    np.testing.assert_array_equal(V, H.f64(vs[0]))


def test_pool_zero_gate_is_window_mean(sk):
    wl = _wl("f32", (0,), (30,), (0,), w=4, H_q=4, H_kv=2, d=64)
    L, (ks, vs, _) = H.gpu_prefill(wl, 0, extra_rows=0, gate_scale=0.0)
    K, _ = L.request_rows(0)
    src = H.f64(ks[0])
    for i in range(8):
        np.testing.assert_allclose(K[i], src[4 * i:4 * i + 4].mean(axis=0), atol=1e-6)


def test_pool_peaked_gate(sk, oracle):
    """Large gate scale: near one-hot window weights stay finite and correct."""
    wl = _wl("bf16", (0,), (64,), (0,), w=8, H_q=16, H_kv=8, d=128)
    L, (ks, vs, gate) = H.gpu_prefill(wl, 0, extra_rows=0, gate_scale=1e3)
    K, V = L.request_rows(0)
    Ko, Vo = oracle.pool_request(H.f64(ks[0]), H.f64(vs[0]), 0, 64, 0, H.f64(gate), 8, 0, 0)
    H.assert_close(K, Ko, "bf16", "K")
    H.assert_close(V, Vo, "bf16", "V")


# --------------------------------------------------------------------------
# append
# --------------------------------------------------------------------------
def test_append_bit_exact_and_capacity(sk, oracle):
    wl = _wl("bf16", (0, 2, 1), (9, 0, 4), (1, 3, 0), w=4, H_q=16, H_kv=8, d=128)
    L, _ = H.gpu_prefill(wl, 0, extra_rows=2)
    lens0 = L.len.cpu().numpy().copy()
    before = [L.request_rows(b) for b in range(wl.B)]
    added_k, added_v = [], []
    for step in range(2):
        _, kn, vn = inputs.step_qkv(wl, 0, step)
        sk.append(kn.cuda(), vn.cuda(), L.k, L.v, L.cache_off, L.len, wl.w, 0, wl.l0)
        added_k.append(H.f64(kn)); added_v.append(H.f64(vn))
        assert (L.len.cpu().numpy() == lens0 + step + 1).all()
        for b in range(wl.B):
            K, V = L.request_rows(b)
            n0 = lens0[b]
            np.testing.assert_array_equal(K[:n0], before[b][0])
            np.testing.assert_array_equal(V[:n0], before[b][1])
            for j in range(step + 1):
                np.testing.assert_array_equal(K[n0 + j], added_k[j][b])
                np.testing.assert_array_equal(V[n0 + j], added_v[j][b])
    assert sk.check_device_error() == sk.OK
    # every cache is now full: a third append writes nothing and reports it
    snap = (L.k.clone(), L.v.clone(), L.len.clone())
    _, kn, vn = inputs.step_qkv(wl, 0, 9)
    sk.append(kn.cuda(), vn.cuda(), L.k, L.v, L.cache_off, L.len, wl.w, 0, wl.l0)
    assert sk.check_device_error() == sk.ERR_CAPACITY
    assert sk.check_device_error() == sk.OK     # cleared by the read
    assert torch.equal(L.k, snap[0]) and torch.equal(L.v, snap[1])
    assert torch.equal(L.len, snap[2])


# --------------------------------------------------------------------------
# decode attention on the GPU's own cache
# --------------------------------------------------------------------------
ATTN_CASES = [
    # dtype, d, H_q, H_kv, P, T, N, G, w
    ("f32", 64, 4, 2, (16,), (64,), (0,), (8,), 4),
    ("f32", 128, 8, 2, (0,), (300,), (7,), (0,), 4),
    ("bf16", 128, 16, 8, (0,), (375,), (32,), (0,), 4),
    ("bf16", 128, 16, 8, (0,), (375,), (32,), (0,), 1),
    ("bf16", 128, 16, 16, (0, 1), (100, 7), (3, 2), (5, 0), 4),   # group 1
    ("bf16", 128, 16, 4, (0,), (500,), (20,), (3,), 8),           # group 4
    ("bf16", 64, 8, 4, (0, 0, 4), (63, 1500, 0), (16, 256, 9), (0, 512, 3), 4),
    ("f32", 64, 16, 4, (2,), (33,), (1,), (0,), 2),
    ("bf16", 128, 6, 3, (0, 2), (200, 50), (10, 4), (3, 0), 4),  # odd H_kv, group 2
    ("bf16", 64, 5, 5, (0,), (120,), (6,), (1,), 4),              # H_kv = 5, group 1
    # tensor-core consumers: 3 to 8 query heads per KV head
    ("bf16", 128, 32, 4, (0, 3), (700, 90), (20, 5), (7, 0), 4),  # group 8
    ("bf16", 64, 32, 4, (0, 0, 4), (63, 1500, 0), (16, 256, 9), (0, 512, 3), 4),  # group 8
    ("bf16", 128, 28, 4, (0, 0), (1200, 31), (40, 2), (5, 1), 4),  # group 7
    ("bf16", 64, 12, 2, (2,), (333,), (7,), (0,), 2),             # group 6
    ("bf16", 128, 20, 4, (1,), (257,), (4,), (0,), 4),            # group 5
    ("bf16", 128, 32, 8, (0,), (500,), (20,), (3,), 1),           # group 4
    ("bf16", 64, 24, 8, (0, 5), (129, 2), (9, 0), (2, 0), 4),     # group 3
]


@pytest.mark.parametrize("dtype,d,H_q,H_kv,P,T,N,G,w", ATTN_CASES)
def test_decode_attn_matches_oracle(sk, oracle, dtype, d, H_q, H_kv, P, T, N, G, w):
    wl = _wl(dtype, P, T, N, G, w=w, H_q=H_q, H_kv=H_kv, d=d)
    L, _ = H.gpu_prefill(wl, 0, extra_rows=0)
    q, _, _ = inputs.step_qkv(wl, 0, 0)
    q = q.cuda()
    ref = _oracle_attn_on_gpu_cache(oracle, wl, L, q)
    for grid in (0, 1, 2, 7, 300):
        out = _decode(sk, wl, L, q, 0, grid=grid)
        H.assert_close(H.f64(out), ref, dtype, f"decode attn, grid {grid}")
    assert sk.check_device_error() == sk.OK


def test_decode_attn_ragged_batch_invariance(sk, oracle):
    """A request's output in a ragged batch matches the same request alone."""
    wl = _wl("bf16", (0,) * 5, (63, 900, 1, 250, 1500), (16, 100, 200, 3, 30),
             (0, 7, 512, 0, 100), w=4, H_q=16, H_kv=8, d=128)
    L, _ = H.gpu_prefill(wl, 0, extra_rows=0)
    q = inputs.step_qkv(wl, 0, 0)[0].cuda()
    full = _decode(sk, wl, L, q, 0)
    for b in (1, 4):
        one = _wl("bf16", (0,), (wl.T[b],), (wl.N[b],), (wl.G[b],), w=4, H_q=16, H_kv=8, d=128)
        L1 = H.GpuLayer(one, 0, 0)
        K, V = L.block(L.k, b), L.block(L.v, b)
        L1.block(L1.k, 0).copy_(K)
        L1.block(L1.v, 0).copy_(V)
        L1.len.copy_(L.len[b:b + 1])
        out1 = _decode(sk, one, L1, q[b:b + 1].contiguous(), 0)
        H.assert_close(H.f64(out1[0]), H.f64(full[b]), "bf16", f"request {b} alone")


def test_decode_attn_edge_cases(sk, oracle):
    wl = _wl("bf16", (0, 0, 0), (8, 16, 4), (0, 2, 0), w=4, H_q=8, H_kv=4, d=128)
    L, _ = H.gpu_prefill(wl, 0, extra_rows=4)
    q = inputs.step_qkv(wl, 0, 0)[0].cuda()
    # an empty request gets zeros; the others are unaffected
    L.len[1] = 0
    out = _decode(sk, wl, L, q, 0)
    assert not out[1].any()
    ref = _oracle_attn_on_gpu_cache(oracle, wl, L, q)
    H.assert_close(H.f64(out), ref, "bf16", "with an empty request")
    # all empty
    L.len.zero_()
    assert not _decode(sk, wl, L, q, 0).any()
    # a length beyond capacity is reported and clamped
    L.len.copy_(torch.tensor([1, 2, 100], dtype=torch.int32))
    out = _decode(sk, wl, L, q, 0)
    assert sk.check_device_error() == sk.ERR_CAPACITY
    L.len[2] = L.cap[2]
    ref = _oracle_attn_on_gpu_cache(oracle, wl, L, q)
    H.assert_close(H.f64(out), ref, "bf16", "clamped length")
    # a single cached row returns its value exactly (up to the output rounding)
    L.len.fill_(1)
    out = _decode(sk, wl, L, q, 0)
    for b in range(wl.B):
        _, V = L.request_rows(b)
        for hq in range(wl.H_q):
            np.testing.assert_array_equal(H.f64(out[b, hq]), V[0, hq // 2])
    # B = 0 is a no-op
    empty = torch.empty((0, 8, 128), dtype=torch.bfloat16, device="cuda")
    sk.decode_attn(empty, L.k, L.v, L.cache_off, L.len[:0], empty, _ws(sk, wl), 4, 0, 0, 4)
    assert sk.check_device_error() == sk.OK


def test_decode_attn_extreme_logits(sk, oracle):
    wl = _wl("bf16", (0,), (600,), (10,), w=4, H_q=16, H_kv=8, d=128)
    L, _ = H.gpu_prefill(wl, 0, extra_rows=0)
    q = (inputs.step_qkv(wl, 0, 0)[0].float() * 100).to(torch.bfloat16).cuda()
    out = _decode(sk, wl, L, q, 0)
    assert torch.isfinite(out.float()).all()
    H.assert_close(H.f64(out), _oracle_attn_on_gpu_cache(oracle, wl, L, q), "bf16", "q x 100")


def test_decode_attn_explicit_scale(sk, oracle):
    wl = _wl("f32", (0,), (100,), (4,), w=4, H_q=4, H_kv=2, d=64)
    L, _ = H.gpu_prefill(wl, 0, extra_rows=0)
    q = inputs.step_qkv(wl, 0, 0)[0].cuda()
    out = _decode(sk, wl, L, q, 0, scale=0.05)
    H.assert_close(H.f64(out), _oracle_attn_on_gpu_cache(oracle, wl, L, q, scale=0.05), "f32",
                   "scale 0.05")


def test_invalid_arguments_return_status(sk):
    wl = _wl("bf16", (0,), (8,), (0,), w=4, H_q=8, H_kv=4, d=128)
    L, _ = H.gpu_prefill(wl, 0, extra_rows=1)
    q = inputs.step_qkv(wl, 0, 0)[0].cuda()
    out = torch.empty_like(q)
    ws = _ws(sk, wl)
    lib = sk.load()
    common = (q.data_ptr(), L.k.data_ptr(), L.v.data_ptr(), L.cache_off.data_ptr(),
              L.len.data_ptr(), out.data_ptr(), 0.0)
    s = torch.cuda.current_stream().cuda_stream
    nbytes = ws.numel()

    def call(B=1, H_q=8, H_kv=4, d=128, w=4, grid=0, wsb=nbytes, dt=sk.BF16, p=common, fl=0):
        return lib.speechkv_decode_attn(*p, B, H_q, H_kv, d, w, 0, 0, grid, ws.data_ptr(), wsb,
                                        dt, fl, s)
    assert call() == sk.OK
    assert call(w=0) == sk.ERR_INVALID_ARG
    assert call(H_q=7) == sk.ERR_INVALID_ARG
    assert call(d=96) == sk.ERR_UNSUPPORTED
    assert call(H_q=64, H_kv=4) == sk.ERR_UNSUPPORTED       # group 16 not built
    assert call(H_q=24, H_kv=8, dt=sk.F32) == sk.ERR_UNSUPPORTED  # fp32: groups 1, 2, 4
    assert call(B=sk.MAX_BATCH + 1) == sk.ERR_UNSUPPORTED
    assert call(wsb=16) == sk.ERR_WORKSPACE
    assert call(grid=-1) == sk.ERR_INVALID_ARG
    assert call(fl=2) == sk.ERR_INVALID_ARG                   # unknown flag
    assert call(fl=sk.OVERLAP_PRIOR) == sk.OK
    misaligned = (q.data_ptr() + 2,) + common[1:]
    assert call(p=misaligned) == sk.ERR_INVALID_ARG
    nullq = (None,) + common[1:]
    assert call(p=nullq) == sk.ERR_INVALID_ARG
    assert sk.check_device_error() == sk.OK


# --------------------------------------------------------------------------
# whole path: prefill pooling, then append + attend for several steps
# --------------------------------------------------------------------------
def _run_steps(sk, oracle, wl, layers, steps, fused=False, grid=0):
    for layer in layers:
        L, (ks, vs, gate) = H.gpu_prefill(wl, layer, extra_rows=steps)
        oc = H.oracle_prefill(oracle, wl, layer, steps, ks, vs, gate)
        ws = _ws(sk, wl, grid)
        store = oracle.STORE_F32 if wl.dtype == "f32" else oracle.STORE_BF16
        for b in range(wl.B):
            assert int(L.len[b]) == oc[b][2]
        for step in range(steps):
            q, kn, vn = inputs.step_qkv(wl, layer, step)
            if fused:
                out = torch.empty_like(q, device="cuda")
                sk.decode_step(q.cuda(), kn.cuda(), vn.cuda(), L.k, L.v, L.cache_off, L.len, out,
                               ws, wl.w, layer, wl.l0, grid_ctas=grid)
            else:
                sk.append(kn.cuda(), vn.cuda(), L.k, L.v, L.cache_off, L.len, wl.w, layer, wl.l0)
                out = _decode(sk, wl, L, q.cuda(), layer, ws=ws, grid=grid)
            ref = []
            for b in range(wl.B):
                Kc, Vc, n = oc[b]
                n = oracle.append_request(Kc, Vc, n, H.f64(kn[b]), H.f64(vn[b]))
                oc[b][2] = n
                assert int(L.len[b]) == n
                ref.append(oracle.decode_attn_request(H.f64(q[b]), Kc[:n], Vc[:n],
                                                      storage=store))
            H.assert_close(H.f64(out), np.stack(ref), wl.dtype, f"layer {layer} step {step}")
    assert sk.check_device_error() == sk.OK


def test_end_to_end_tiny_fp32(sk, oracle):
    """Tiny fp32 workload: 16 text + 64 frames (w=4 -> 16 entries), 8 steps;
    cached rows go 33 -> 40."""
    _run_steps(sk, oracle, inputs.tiny_fp32(), layers=[0], steps=8)


def test_end_to_end_qwen_single(sk, oracle):
    """Qwen3-1.7B shapes, 30 s audio: one layer before l0 (full resolution)
    and one pooled layer, first 6 of the 128 steps."""
    wl = inputs.qwen_single()
    _run_steps(sk, oracle, wl, layers=[wl.l0 - 1, wl.l0], steps=6)


def test_end_to_end_ragged_small(sk, oracle):
    wl = inputs.qwen_ragged(B=6)
    _run_steps(sk, oracle, wl, layers=[wl.l0], steps=3)


def test_per_layer_windows(sk, oracle):
    """Compression ratios that differ across layers (the paper leaves adaptive
    ratios to future work): the window is an argument of every call, so each
    layer's cache may be pooled with its own w.  Layers 7 (before l0), 8, 9, 10
    with w = 4 (unused: full resolution), 2, 4, 8; fused decode steps."""
    base = inputs.qwen_single()
    for layer, w in ((base.l0 - 1, 4), (base.l0, 2), (base.l0 + 1, 4), (base.l0 + 2, 8)):
        _run_steps(sk, oracle, dataclasses.replace(base, w=w), layers=[layer], steps=3, fused=True)


# --------------------------------------------------------------------------
# fused step: append + decode attention in one launch
# --------------------------------------------------------------------------
@pytest.mark.parametrize("grid", [0, 1, 7, 300])
def test_fused_step_tiny_fp32(sk, oracle, grid):
    _run_steps(sk, oracle, inputs.tiny_fp32(), layers=[0], steps=8, fused=True, grid=grid)


def test_fused_step_qwen_and_ragged(sk, oracle):
    wl = inputs.qwen_single()
    _run_steps(sk, oracle, wl, layers=[wl.l0 - 1, wl.l0], steps=4, fused=True)
    wl = inputs.qwen_ragged(B=6)
    _run_steps(sk, oracle, wl, layers=[wl.l0], steps=3, fused=True)


@pytest.mark.parametrize("H_q,H_kv", [(32, 4), (28, 4), (24, 8)])
def test_fused_step_groups_3_to_8(sk, oracle, H_q, H_kv):
    """Fused steps with the tensor-core consumers (8, 7 and 3 query heads per
    KV head) on a ragged batch, from the oracle's pooling on."""
    wl = dataclasses.replace(inputs.qwen_ragged(B=6), H_q=H_q, H_kv=H_kv)
    _run_steps(sk, oracle, wl, layers=[wl.l0 - 1, wl.l0], steps=3, fused=True)


def test_fused_step_matches_separate_calls_and_writes_cache(sk):
    """decode_step leaves the same cache and lengths as append + decode_attn
    (bit-exact) and gives the same output up to summation order."""
    wl = _wl("bf16", (0, 0, 3), (375, 40, 9), (32, 5, 0), (3, 0, 1), w=4, H_q=16, H_kv=8,
             d=128)
    A, _ = H.gpu_prefill(wl, 0, extra_rows=3)
    Bc, _ = H.gpu_prefill(wl, 0, extra_rows=3)
    wsA, wsB = _ws(sk, wl), _ws(sk, wl)
    for step in range(3):
        q, kn, vn = (x.cuda() for x in inputs.step_qkv(wl, 0, step))
        sk.append(kn, vn, A.k, A.v, A.cache_off, A.len, wl.w, 0, wl.l0)
        outA = _decode(sk, wl, A, q, 0, ws=wsA)
        outB = torch.empty_like(q)
        sk.decode_step(q, kn, vn, Bc.k, Bc.v, Bc.cache_off, Bc.len, outB, wsB, wl.w, 0, wl.l0)
        assert torch.equal(A.len, Bc.len)
        assert torch.equal(A.k, Bc.k) and torch.equal(A.v, Bc.v)
        H.assert_close(H.f64(outB), H.f64(outA), "bf16", f"step {step}")
    assert sk.check_device_error() == sk.OK


@pytest.mark.parametrize("graph", [False, True])
def test_overlap_prior_interleaved_layers(sk, oracle, graph):
    """SPEECHKV_OVERLAP_PRIOR between the decode steps of different layers
    (the previous kernel writes another layer's cache, its length and the
    shared workspace): results still match the oracle, eagerly and when the
    steps are captured in a CUDA graph."""
    wl = inputs.qwen_ragged(B=5)
    layers, steps = [wl.l0 - 1, wl.l0, wl.l0 + 1], 3
    gl, ol = [], []
    for layer in layers:
        L, (ks, vs, gate) = H.gpu_prefill(wl, layer, extra_rows=steps)
        gl.append(L)
        ol.append(H.oracle_prefill(oracle, wl, layer, steps, ks, vs, gate))
    ws = _ws(sk, wl)
    ins = [[[x.cuda() for x in inputs.step_qkv(wl, layer, t)] for layer in layers]
           for t in range(steps)]
    outs = [[torch.empty_like(ins[0][0][0]) for _ in layers] for _ in range(steps)]

    def run():
        for t in range(steps):
            for i, layer in enumerate(layers):
                q, kn, vn = ins[t][i]
                L = gl[i]
                sk.decode_step(q, kn, vn, L.k, L.v, L.cache_off, L.len, outs[t][i], ws, wl.w,
                               layer, wl.l0, flags=sk.OVERLAP_PRIOR)
    if graph:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            run()
        g.replay()
    else:
        run()
    torch.cuda.synchronize()
    assert sk.check_device_error() == sk.OK
    for t in range(steps):
        for i, layer in enumerate(layers):
            q, kn, vn = (x.cpu() for x in ins[t][i])
            ref = []
            for b in range(wl.B):
                Kc, Vc, n = ol[i][b]
                n = oracle.append_request(Kc, Vc, n, H.f64(kn[b]), H.f64(vn[b]))
                ol[i][b][2] = n
                ref.append(oracle.decode_attn_request(H.f64(q[b]), Kc[:n], Vc[:n],
                                                      storage=oracle.STORE_BF16))
            H.assert_close(H.f64(outs[t][i]), np.stack(ref), "bf16", f"step {t} layer {layer}")
    for i in range(len(layers)):
        assert [int(x) for x in gl[i].len.cpu()] == [o[2] for o in ol[i]]


def test_fused_step_full_cache(sk, oracle):
    """A full cache takes no token: CAPACITY is reported, len stays, and the
    output is attention over the cached rows alone."""
    wl = _wl("bf16", (0, 0), (20, 12), (2, 3), w=4, H_q=8, H_kv=4, d=128)
    L, _ = H.gpu_prefill(wl, 0, extra_rows=0)       # capacity == rows: full
    q, kn, vn = (x.cuda() for x in inputs.step_qkv(wl, 0, 0))
    lens, kbefore = L.len.clone(), L.k.clone()
    out = torch.empty_like(q)
    sk.decode_step(q, kn, vn, L.k, L.v, L.cache_off, L.len, out, _ws(sk, wl), wl.w, 0, wl.l0)
    assert sk.check_device_error() == sk.ERR_CAPACITY
    assert torch.equal(L.len, lens) and torch.equal(L.k, kbefore)
    H.assert_close(H.f64(out), _oracle_attn_on_gpu_cache(oracle, wl, L, q), "bf16", "full")


# --------------------------------------------------------------------------
# full benchmark sizes, sampled against the oracle
# --------------------------------------------------------------------------
def _sampled_full_size(sk, oracle, wl, layer, samples, fused=False):
    L, _ = H.gpu_prefill(wl, layer, extra_rows=1)
    q, kn, vn = inputs.step_qkv(wl, layer, 0)
    if fused:
        out = torch.empty_like(q, device="cuda")
        sk.decode_step(q.cuda(), kn.cuda(), vn.cuda(), L.k, L.v, L.cache_off, L.len, out,
                       _ws(sk, wl), wl.w, layer, wl.l0)
    else:
        sk.append(kn.cuda(), vn.cuda(), L.k, L.v, L.cache_off, L.len, wl.w, layer, wl.l0)
        out = _decode(sk, wl, L, q.cuda(), layer)
    assert sk.check_device_error() == sk.OK
    lens = L.len.cpu().numpy()
    for b in samples:
        assert lens[b] == oracle.compressed_len(wl.P[b], wl.T[b], wl.N[b], wl.G[b] + 1, wl.w,
                                                layer, wl.l0)
        K, V = L.request_rows(b)
        ref = oracle.decode_attn_request(H.f64(q[b]), K, V, storage=oracle.STORE_BF16)
        H.assert_close(H.f64(out[b]), ref, "bf16", f"request {b}")


@pytest.mark.parametrize("minutes,w", [(20, 4), (10, 8)])
def test_full_size_long_audio_sampled(sk, oracle, minutes, w):
    wl = inputs.qwen_long_audio(minutes, w, generated=64)
    _sampled_full_size(sk, oracle, wl, wl.l0, samples=[0, 5])


@pytest.mark.parametrize("fused", [False, True])
def test_full_size_ragged_sampled(sk, oracle, fused):
    wl = inputs.qwen_ragged()
    _sampled_full_size(sk, oracle, wl, wl.l0, samples=[0, 17, 64, 127], fused=fused)


@pytest.mark.parametrize("H_q,H_kv", [(32, 8), (32, 4), (28, 4)])
def test_full_size_long_audio_groups(sk, oracle, H_q, H_kv):
    """The 20 min / w = 4 batch with 4, 8 and 7 query heads per KV head
    (tensor-core consumers), fused step, sampled requests."""
    wl = dataclasses.replace(inputs.qwen_long_audio(20, 4, generated=64), H_q=H_q, H_kv=H_kv)
    _sampled_full_size(sk, oracle, wl, wl.l0, samples=[1, 6], fused=True)


def test_full_size_long_audio_fused(sk, oracle):
    wl = inputs.qwen_long_audio(20, 4, generated=64)
    _sampled_full_size(sk, oracle, wl, wl.l0, samples=[3], fused=True)


@pytest.mark.parametrize("H_q,H_kv", [(16, 8), (32, 4)])
def test_max_batch_fused_step(sk, oracle, H_q, H_kv):
    """B = SPEECHKV_MAX_BATCH (the largest per-request tables in shared
    memory), short random lengths: pooling, one fused decode step, sampled
    requests against the oracle (2 and 8 query heads per KV head: the
    8-head instance has the largest merge buffers)."""
    rng = np.random.default_rng(4242)
    B = sk.MAX_BATCH
    T = [int(x) for x in rng.integers(1, 60, B)]
    N = [int(x) for x in rng.integers(0, 20, B)]
    wl = inputs.Workload(name="maxbatch", dtype="bf16", L=28, l0=8, w=4, H_q=H_q, H_kv=H_kv,
                         d=128, P=[0] * B, T=T, N=N, G=[0] * B, steps=1, seed=4242)
    layer = wl.l0
    L, (ks, vs, gate) = H.gpu_prefill(wl, layer, extra_rows=1)
    ws = sk.new_workspace(wl.B, wl.H_q, wl.H_kv, wl.d)
    q, kn, vn = inputs.step_qkv(wl, layer, 0)
    out = torch.empty_like(q, device="cuda")
    sk.decode_step(q.cuda(), kn.cuda(), vn.cuda(), L.k, L.v, L.cache_off, L.len, out, ws, wl.w,
                   layer, wl.l0)
    assert sk.check_device_error() == sk.OK
    for b in sorted(set([0, 1, B - 1] + [int(x) for x in rng.integers(0, B, 13)])):
        Ko, Vo = oracle.pool_request(H.f64(ks[b]), H.f64(vs[b]), 0, T[b], N[b], H.f64(gate),
                                     wl.w, layer, wl.l0, storage=oracle.STORE_BF16)
        n = Ko.shape[0]
        Kc = np.zeros((n + 1, wl.H_kv, wl.d)); Vc = np.zeros_like(Kc)
        Kc[:n], Vc[:n] = Ko, Vo
        n = oracle.append_request(Kc, Vc, n, H.f64(kn[b]), H.f64(vn[b]))
        assert int(L.len[b]) == n
        ref = oracle.decode_attn_request(H.f64(q[b]), Kc[:n], Vc[:n], storage=oracle.STORE_BF16)
        H.assert_close(H.f64(out[b]), ref, "bf16", f"request {b}")


@pytest.mark.parametrize("grid,H_kv", [(0, 8), (7, 8), (16, 8), (0, 4), (7, 4), (7, 16),
                                     (0, 2), (7, 2)])
def test_overlap_prior_two_layer_interleave_any_grid(sk, oracle, grid, H_kv):
    """SPEECHKV_OVERLAP_PRIOR with the steps of two layers interleaved
    [a, b, a, b, ...]: the kernel two launches back writes this call's cache
    and length.  A decode kernel releases its successor only after its own
    wait for its predecessor, so that kernel has completed before this one
    starts, whatever the grid -- small explicit grids, under which several
    grids fit on the GPU at once, included."""
    # H_kv 4 / 16 with 16 query heads: groups of 4 (a two-stage ring) and 1
    wl = dataclasses.replace(inputs.qwen_ragged(B=5), H_kv=H_kv)
    layers, steps = [wl.l0 - 1, wl.l0], 4
    gl, ol = [], []
    for layer in layers:
        L, (ks, vs, gate) = H.gpu_prefill(wl, layer, extra_rows=steps)
        gl.append(L)
        ol.append(H.oracle_prefill(oracle, wl, layer, steps, ks, vs, gate))
    ws = _ws(sk, wl, grid)
    ins = [[[x.cuda() for x in inputs.step_qkv(wl, layer, t)] for layer in layers]
           for t in range(steps)]
    outs = [[torch.empty_like(ins[0][0][0]) for _ in layers] for _ in range(steps)]
    for t in range(steps):
        for i, layer in enumerate(layers):
            q, kn, vn = ins[t][i]
            L = gl[i]
            sk.decode_step(q, kn, vn, L.k, L.v, L.cache_off, L.len, outs[t][i], ws, wl.w, layer,
                           wl.l0, grid_ctas=grid, flags=sk.OVERLAP_PRIOR)
    torch.cuda.synchronize()
    assert sk.check_device_error() == sk.OK
    for t in range(steps):
        for i, layer in enumerate(layers):
            q, kn, vn = (x.cpu() for x in ins[t][i])
            ref = []
            for b in range(wl.B):
                Kc, Vc, n = ol[i][b]
                n = oracle.append_request(Kc, Vc, n, H.f64(kn[b]), H.f64(vn[b]))
                ol[i][b][2] = n
                ref.append(oracle.decode_attn_request(H.f64(q[b]), Kc[:n], Vc[:n],
                                                      storage=oracle.STORE_BF16))
            H.assert_close(H.f64(outs[t][i]), np.stack(ref), "bf16",
                           f"grid {grid} step {t} layer {layer}")
    for i in range(len(layers)):
        assert [int(x) for x in gl[i].len.cpu()] == [o[2] for o in ol[i]]
        # every appended row sits where the oracle put it (no row written twice)
        for b in range(wl.B):
            K, V = gl[i].request_rows(b)
            Kc, Vc, n = ol[i][b]
            np.testing.assert_array_equal(K[n - steps:], Kc[n - steps:n])
            np.testing.assert_array_equal(V[n - steps:], Vc[n - steps:n])


# --------------------------------------------------------------------------
# pooling at the long-audio benchmark's full size, element by element
# --------------------------------------------------------------------------
@pytest.mark.parametrize("minutes,w,T", [(20, 4, None), (20, 4, 14999), (10, 8, None)])
def test_pool_full_size_matches_oracle(sk, oracle, minutes, w, T):
    """The pooled layer l0 of the long-audio batch (8 requests; 20 min is
    15,000 frames, with a 14,999-frame variant whose last window holds three
    frames), every row of every KV head of the first and the last request
    against Eq. (pool) in the oracle.  Text rows are bit-exact copies."""
    wl = inputs.qwen_long_audio(minutes, w)
    if T is not None:
        wl = dataclasses.replace(wl, T=[T] * wl.B)
    layer = wl.l0
    L, (ks, vs, gate) = H.gpu_prefill(wl, layer, extra_rows=1)
    assert sk.check_device_error() == sk.OK
    lens = L.len.cpu().numpy()
    for b in range(wl.B):
        assert lens[b] == oracle.compressed_len(wl.P[b], wl.T[b], wl.N[b], 0, w, layer, wl.l0)
    for b in (0, wl.B - 1):
        Ko, Vo = oracle.pool_request(H.f64(ks[b]), H.f64(vs[b]), wl.P[b], wl.T[b], wl.N[b],
                                     H.f64(gate), w, layer, wl.l0, storage=oracle.STORE_BF16)
        K, V = L.request_rows(b)
        H.assert_close(K, Ko, "bf16", f"pooled K, request {b}")
        H.assert_close(V, Vo, "bf16", f"pooled V, request {b}")
        n = Ko.shape[0] - wl.P[b] - wl.N[b]
        # the first, a middle and the last (possibly partial) window, tighter:
        # one rounding to bf16 of the fp32 result
        for i in (0, n // 2, n - 1):
            np.testing.assert_allclose(K[wl.P[b] + i], Ko[wl.P[b] + i], rtol=2 ** -7, atol=1e-6)
            np.testing.assert_allclose(V[wl.P[b] + i], Vo[wl.P[b] + i], rtol=2 ** -7, atol=1e-6)
        src_k, src_v = H.f64(ks[b]), H.f64(vs[b])
        np.testing.assert_array_equal(K[wl.P[b] + n:], src_k[wl.P[b] + wl.T[b]:])
        np.testing.assert_array_equal(V[wl.P[b] + n:], src_v[wl.P[b] + wl.T[b]:])


# --------------------------------------------------------------------------
# batch of 64 uniform 30 s requests, compressed and uncompressed
# --------------------------------------------------------------------------
@pytest.mark.parametrize("w", [4, 1])
def test_batch64_30s_pool_and_fused_steps(sk, oracle, w):
    """64 requests of 30 s audio (375 frames) and a 32-token prompt at
    Qwen3-1.7B shapes, pooled with w = 4 from l0 = 8 and its uncompressed
    twin (w = 1, identical seeded tensors): pooling, then three fused decode
    steps at layers l0 - 1 and l0, every request against the oracle's
    pooling -> appends -> attention."""
    wl = inputs.qwen_batch64(w=w)
    _run_steps(sk, oracle, wl, layers=[wl.l0 - 1, wl.l0], steps=3, fused=True)


@pytest.mark.parametrize("H_kv,grid", [(8, 0), (8, 1), (8, 3), (4, 0), (4, 5), (16, 0), (16, 2),
                                     (2, 0), (2, 3)])
def test_short_requests_share_tiles(sk, oracle, H_kv, grid):
    """Many short requests (0-20 rows, some empty) so that a 128-row tile
    holds the ends and starts of several (request, KV head) runs: tiles are
    cut before a third run would start in them, and pieces of one row occur.
    Fused steps against the oracle's pooling -> append -> attention."""
    rng = np.random.default_rng(77 + H_kv + grid)
    B = 40
    T = [int(x) for x in rng.integers(0, 12, B)]
    N = [int(x) for x in rng.integers(0, 9, B)]
    T[3] = N[3] = 0                      # an empty request (its rows come from the steps)
    wl = inputs.Workload(name="short", dtype="bf16", L=1, l0=0, w=4, H_q=16, H_kv=H_kv, d=128,
                         P=[0] * B, T=T, N=N, G=[0] * B, steps=2, seed=78)
    _run_steps(sk, oracle, wl, layers=[0], steps=2, fused=True, grid=grid)
