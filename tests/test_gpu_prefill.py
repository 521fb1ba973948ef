"""GPU parity of speechkv_prefill_attn -- Eq. (attn) at prefill with the
adjusted causal mask (Sec. III-B) -- against the CPU oracle.

The kernel runs on tensor cores with bf16 operands and bf16 softmax weights
in the P V product; the bf16 tolerances (max-abs 2e-2, mean-abs 2e-3 on
unit-variance inputs) apply.  Every case checks the kernel on the GPU's own
pooled cache (isolating the attention), most also end to end from the same
full-resolution prompt through the oracle's pooling."""
import itertools

import numpy as np
import pytest
import torch

from paper_2607_06827_gb300 import inputs
from tests import harness as H

pytestmark = pytest.mark.gpu


def _wl(P, T, N, w=4, l0=8, seed=2001, H_q=16, H_kv=8, d=128):
    return inputs.Workload(name="prefill", dtype="bf16", L=28, l0=l0, w=w, H_q=H_q, H_kv=H_kv,
                           d=d, P=list(P), T=list(T), N=list(N), G=[0] * len(T), steps=0,
                           seed=seed)


def _q_off(wl):
    off = np.zeros(wl.B + 1, dtype=np.int64)
    off[1:] = np.cumsum(wl.full_rows())
    return off


def _run(wl, layer, pad_rows=0, sentinel=7.0):
    """Pool the prompt on the GPU, then run the prefill attention over it."""
    H.require_gpu()
    sk = H.lib()
    L, full = H.gpu_prefill(wl, layer, extra_rows=0)
    qs = [inputs.prefill_q(wl, layer, b) for b in range(wl.B)]
    q = torch.cat(qs).cuda()
    if pad_rows:
        q = torch.cat([q, torch.randn(pad_rows, wl.H_q, wl.d, device="cuda").to(q.dtype)])
    out = torch.full_like(q, sentinel)
    P, T, N = H.lengths_dev(wl)
    q_off = torch.from_numpy(_q_off(wl)).cuda()
    sk.prefill_attn(q, q_off, P, T, N, L.k, L.v, L.cache_off, out, wl.w, layer, wl.l0, wl.H_kv)
    assert sk.check_device_error() == sk.OK
    return L, qs, out, full


def _w_eff(wl, layer):
    return wl.w if layer >= wl.l0 else 1


def _check(oracle, wl, layer, L, qs, out, full=None):
    off = _q_off(wl)
    ends = H.oracle_prefill(oracle, wl, layer, 0, *full) if full is not None else None
    for b in range(wl.B):
        c = int(L.len[b].item())
        got = H.f64(out[off[b]:off[b + 1]])
        K, V = L.request_rows(b, c)
        ref = oracle.prefill_attn_request(H.f64(qs[b]), K, V, wl.P[b], wl.T[b], wl.N[b],
                                          _w_eff(wl, layer), storage=oracle.STORE_BF16)
        H.assert_close(got, ref, "bf16", f"request {b} on the GPU's cache")
        if ends is not None:
            Kc, Vc, n = ends[b]
            assert n == c
            ref2 = oracle.prefill_attn_request(H.f64(qs[b]), Kc[:n], Vc[:n], wl.P[b], wl.T[b],
                                               wl.N[b], _w_eff(wl, layer),
                                               storage=oracle.STORE_BF16)
            H.assert_close(got, ref2, "bf16", f"request {b} end to end")


@pytest.mark.parametrize("layer,d", [(8, 128), (0, 128), (8, 64), (0, 64)])
def test_prefill_matches_oracle(oracle, layer, d):
    """A pooled layer (w = 4) and a full-resolution one (causal attention);
    ragged requests: speech only with text after, a text prefix, text only;
    head dimensions 128 and 64."""
    wl = _wl(P=[0, 16, 5], T=[375, 130, 0], N=[32, 7, 40], d=d)
    L, qs, out, full = _run(wl, layer)
    _check(oracle, wl, layer, L, qs, out, full)


@pytest.mark.parametrize("d", [128, 64])
@pytest.mark.parametrize("P,T,N,w", [
    ([0, 0, 0, 3], [1, 128, 512, 1], [0, 0, 1, 0], 4),     # one row, exact tiles, S = 129
    ([0, 7], [255, 1000], [1, 3], 8),                      # w = 8, several key tiles
    ([130, 0], [0, 513], [0, 200], 3),                     # text only; w = 3 (tiles cut windows)
])
def test_prefill_edge_lengths(oracle, P, T, N, w, d):
    wl = _wl(P, T, N, w=w, seed=2002, d=d)
    L, qs, out, full = _run(wl, 8)
    _check(oracle, wl, 8, L, qs, out, full)


def test_prefill_gqa_groups(oracle):
    """Query heads per KV head 1, 3 and 4 (the head mapping hq / group).  A
    work item holds up to two query heads of one KV head: with one head per
    KV head the second tile of every item is idle, with three the items
    alternate between two heads and one."""
    for (H_q, H_kv), d in itertools.product(((8, 8), (12, 4), (16, 4)), (128, 64)):
        wl = _wl(P=[4], T=[300], N=[20], H_q=H_q, H_kv=H_kv, seed=2003, d=d)
        L, qs, out, full = _run(wl, 8)
        _check(oracle, wl, 8, L, qs, out)


def test_prefill_leaves_other_rows_alone():
    """Rows of q / out past the last request are neither read into any
    output nor written."""
    wl = _wl(P=[0, 2], T=[200, 60], N=[10, 0], seed=2004)
    L, qs, out, _ = _run(wl, 8, pad_rows=77, sentinel=7.0)
    S = sum(wl.full_rows())
    assert torch.all(out[S:] == 7.0)
    assert torch.isfinite(out[:S].float()).all()
    assert not torch.any(out[:S] == 7.0)


def test_prefill_batch_invariance():
    """Each request's rows are the same whether it runs alone or in a batch
    (a request's result does not depend on the others)."""
    H.require_gpu()
    sk = H.lib()
    wl = _wl(P=[0, 16, 5], T=[375, 130, 33], N=[32, 7, 40], seed=2005)
    layer = 8
    L, qs, out, _ = _run(wl, layer)
    off = _q_off(wl)
    for b in range(wl.B):
        one = _wl([wl.P[b]], [wl.T[b]], [wl.N[b]], seed=2005)
        # the single request gets the same cache rows and queries
        Lb = H.GpuLayer(one, layer, 0)
        c = int(L.len[b].item())
        Lb.block(Lb.k, 0)[:, :c] = L.block(L.k, b)[:, :c]
        Lb.block(Lb.v, 0)[:, :c] = L.block(L.v, b)[:, :c]
        qb = qs[b].cuda()
        ob = torch.zeros_like(qb)
        P, T, N = H.lengths_dev(one)
        q_off = torch.tensor([0, qb.shape[0]], dtype=torch.int64, device="cuda")
        sk.prefill_attn(qb, q_off, P, T, N, Lb.k, Lb.v, Lb.cache_off, ob, one.w, layer, one.l0,
                        one.H_kv)
        assert sk.check_device_error() == sk.OK
        assert torch.equal(ob, out[off[b]:off[b + 1]])


def test_prefill_inconsistent_rows_are_reported():
    """A request whose query rows disagree with P + T + N is skipped and
    reported as an invalid argument (no fault, the others still run)."""
    H.require_gpu()
    sk = H.lib()
    wl = _wl(P=[0, 0], T=[100, 100], N=[4, 4], seed=2006)
    L, qs, out, _ = _run(wl, 8)
    q = torch.cat(qs).cuda()
    bad = torch.full_like(q, 3.0)
    P, T, N = H.lengths_dev(wl)
    q_off = torch.tensor([0, 104, 200], dtype=torch.int64, device="cuda")  # request 1: 96 != 104
    sk.prefill_attn(q, q_off, P, T, N, L.k, L.v, L.cache_off, bad, wl.w, 8, wl.l0, wl.H_kv)
    assert sk.check_device_error() == sk.ERR_INVALID_ARG
    assert torch.equal(bad[:104], out[:104])   # request 0 computed as before
    assert torch.all(bad[104:] == 3.0)         # request 1 skipped


def test_prefill_full_size_sampled(oracle):
    """The 20 min / batch 8 prompt at a pooled layer, as the bench runs it;
    sampled rows against the oracle.  A prefill row attends over exactly the
    cache prefix 0 .. pi(t), so its reference is the decode attention of that
    query over that prefix."""
    H.require_gpu()
    sk = H.lib()
    wl = inputs.qwen_long_audio(20, 4)
    layer = wl.l0
    L = H.GpuLayer(wl, layer, 0)
    c = [sk.compressed_len(wl.P[b], wl.T[b], wl.N[b], 0, wl.w, layer, wl.l0) for b in range(wl.B)]
    L.k.copy_(inputs.device_normal(L.k.shape, L.k.dtype, "cuda", wl.seed, 30, layer))
    L.v.copy_(inputs.device_normal(L.v.shape, L.v.dtype, "cuda", wl.seed, 31, layer))
    L.len.copy_(torch.tensor(c, dtype=torch.int32))
    S = sum(wl.full_rows())
    q = inputs.device_normal((S, wl.H_q, wl.d), torch.bfloat16, "cuda", wl.seed, 32, layer)
    out = torch.zeros_like(q)
    P, T, N = H.lengths_dev(wl)
    off = _q_off(wl)
    sk.prefill_attn(q, torch.from_numpy(off).cuda(), P, T, N, L.k, L.v, L.cache_off, out, wl.w,
                    layer, wl.l0, wl.H_kv)
    assert sk.check_device_error() == sk.OK
    rng = np.random.default_rng(7)
    for b in (0, 3, 7):
        Sb = wl.full_rows()[b]
        K, V = L.request_rows(b, c[b])
        rows = sorted(set([0, 1, 127, 128, 5000, Sb - 65, Sb - 1] +
                          list(rng.integers(0, Sb, 5))))
        for t in rows:
            last = oracle.prefill_position(wl.P[b], wl.T[b], wl.N[b], wl.w, int(t))
            qt = H.f64(q[off[b] + t])
            ref = oracle.decode_attn_request(qt, K[:last + 1], V[:last + 1],
                                             storage=oracle.STORE_BF16)
            H.assert_close(H.f64(out[off[b] + t]), ref, "bf16", f"request {b} row {t}")


def test_prefill_random_shapes(oracle):
    """Seeded random batches: 1-6 requests with random text and speech
    lengths, windows 1-8, several query/KV head ratios, pooled and
    full-resolution layers; every request against the oracle on the GPU's
    cache, and three launches bit-identical."""
    H.require_gpu()
    sk = H.lib()
    rng = np.random.default_rng(2007)
    heads = [(2, 2), (6, 2), (8, 8), (12, 4), (16, 8)]
    for case in range(12):
        B = int(rng.integers(1, 7))
        H_q, H_kv = heads[int(rng.integers(len(heads)))]
        w = int(rng.choice([1, 2, 3, 4, 5, 8]))
        P = [int(x) for x in rng.integers(0, 40, B)]
        T = [int(x) for x in rng.integers(0, 500, B)]
        N = [max(int(x), 1 if p + t == 0 else 0) for x, p, t in zip(rng.integers(0, 80, B), P, T)]
        layer = int(rng.choice([0, 8]))
        d = int(rng.choice([64, 128]))
        wl = _wl(P, T, N, w=w, seed=2100 + case, H_q=H_q, H_kv=H_kv, d=d)
        L, full = H.gpu_prefill(wl, layer, extra_rows=int(rng.integers(0, 4)))
        qs = [inputs.prefill_q(wl, layer, b) for b in range(wl.B)]
        q = torch.cat(qs).cuda()
        Pd, Td, Nd = H.lengths_dev(wl)
        q_off = torch.from_numpy(_q_off(wl)).cuda()
        outs = []
        for _ in range(3):
            out = torch.full_like(q, 3.0)
            sk.prefill_attn(q, q_off, Pd, Td, Nd, L.k, L.v, L.cache_off, out, w, layer, wl.l0,
                            H_kv)
            assert sk.check_device_error() == sk.OK
            outs.append(out)
        assert all(torch.equal(outs[0], o) for o in outs[1:]), f"case {case}: not deterministic"
        _check(oracle, wl, layer, L, qs, outs[0])


def test_prefill_max_batch(oracle):
    """B = SPEECHKV_MAX_BATCH requests with short random lengths (many small
    items, the request table read per item), every request against the
    oracle."""
    H.require_gpu()
    sk = H.lib()
    rng = np.random.default_rng(2011)
    B = sk.MAX_BATCH
    T = [int(x) for x in rng.integers(0, 200, B)]
    N = [int(x) for x in rng.integers(1, 40, B)]
    P = [int(x) for x in rng.integers(0, 8, B)]
    wl = _wl(P, T, N, w=4, seed=2011)
    L, qs, out, full = _run(wl, 8)
    _check(oracle, wl, 8, L, qs, out)
