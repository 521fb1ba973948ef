"""GPU tests of the paged cache layout (block tables, as in the paper's
serving system): speechkv_pool_paged, speechkv_append_paged,
speechkv_decode_step_paged and speechkv_prefill_attn_paged against the
contiguous entry points on the same inputs.
Paging only moves rows: caches and lengths must be bit-identical, and so
must the fp32 decode outputs and the prefill outputs; bf16 decode outputs
are equal up to summation order (over a block table the decode tiles start
on 16-row boundaries).  One case is also checked against the oracle
directly."""
import dataclasses

import numpy as np
import pytest
import torch

from paper_2607_06827_gb300 import inputs
from tests import harness as H

pytestmark = pytest.mark.gpu


class Paged:
    """One layer's pages with a shuffled block table (seeded)."""

    def __init__(self, wl, layer, extra_rows, block_size, seed=0, spare=3):
        sk = H.lib()
        self.wl, self.bs = wl, block_size
        cap = [sk.compressed_len(p, t, n, g, wl.w, layer, wl.l0) + extra_rows
               for p, t, n, g in zip(wl.P, wl.T, wl.N, wl.G)]
        self.max_blocks = max(-(-c // block_size) for c in cap)
        need = [-(-c // block_size) for c in cap]
        self.num_blocks = sum(need) + spare
        perm = np.random.default_rng(seed).permutation(self.num_blocks)
        table = np.full((wl.B, self.max_blocks), -1, dtype=np.int32)
        k = 0
        for b in range(wl.B):
            table[b, :need[b]] = perm[k:k + need[b]]
            k += need[b]
        self.table = torch.from_numpy(table).cuda()
        shape = (self.num_blocks, wl.H_kv, block_size, wl.d)
        dt = H.TORCH_DTYPE[wl.dtype]
        self.k = torch.full(shape, 9.0, dtype=dt, device="cuda")
        self.v = torch.full(shape, 9.0, dtype=dt, device="cuda")
        self.len = torch.zeros(wl.B, dtype=torch.int32, device="cuda")

    def rows(self, t, b, n):
        """Request b's first n rows of a page tensor as [H_kv, n, d]."""
        table = self.table.cpu().numpy()
        idx = [int(table[b, r // self.bs]) for r in range(n)]
        slot = [r % self.bs for r in range(n)]
        return t[idx, :, slot, :].permute(1, 0, 2) if n else t[:0, :, 0, :].permute(1, 0, 2)


def _prefill_both(wl, layer, extra, block_size, seed=0):
    sk = H.lib()
    L, (ks, vs, gate) = H.gpu_prefill(wl, layer, extra_rows=extra)
    pg = Paged(wl, layer, extra, block_size, seed)
    k, v, full_off, _, _ = H.prefill_packed(wl, layer)
    P, T, N = H.lengths_dev(wl)
    g = torch.from_numpy(inputs.gate(wl, layer)).cuda()
    sk.pool_paged(k, v, full_off, P, T, N, g, pg.k, pg.v, pg.table, pg.len, wl.w, layer, wl.l0)
    assert sk.check_device_error() == sk.OK
    return L, pg, (ks, vs, gate)


def _same_cache(wl, L, pg):
    assert torch.equal(L.len, pg.len)
    for b in range(wl.B):
        n = int(L.len[b])
        assert torch.equal(L.block(L.k, b)[:, :n], pg.rows(pg.k, b, n)), f"keys of request {b}"
        assert torch.equal(L.block(L.v, b)[:, :n], pg.rows(pg.v, b, n)), f"values of request {b}"


@pytest.mark.parametrize("block_size,H_kv", [(16, 8), (64, 8), (128, 8), (256, 8), (16, 2),
                                            (64, 2), (8, 4)])
def test_paged_steps_match_contiguous(block_size, H_kv):
    """Pooling, generated-token appends and fused decode steps at a pooled
    layer, ragged batch (16 query heads over 8, 2 or 4 KV heads): the caches
    bit-identical to the contiguous path's, the outputs equal up to summation
    order (over a block table the tiles start on 16-row boundaries, so the
    rows fall to other warps than in a contiguous cache)."""
    sk = H.lib()
    wl = inputs.qwen_ragged(B=6)
    wl = dataclasses.replace(wl, G=[0] * wl.B, H_kv=H_kv)  # history from the appends below
    layer, steps, G = wl.l0, 4, 3
    L, pg, _ = _prefill_both(wl, layer, steps + G, block_size, seed=block_size)
    _same_cache(wl, L, pg)
    ws = sk.new_workspace(wl.B, wl.H_q, wl.H_kv, wl.d)
    ws2 = sk.new_workspace(wl.B, wl.H_q, wl.H_kv, wl.d)
    for step in range(G):  # tokens generated before the checked steps
        kn, vn = (inputs.device_normal((wl.B, wl.H_kv, wl.d), torch.bfloat16, "cuda", 7, step, x)
                  for x in (1, 2))
        sk.append(kn, vn, L.k, L.v, L.cache_off, L.len, wl.w, layer, wl.l0)
        sk.append_paged(kn, vn, pg.k, pg.v, pg.table, pg.len, wl.w, layer, wl.l0)
    _same_cache(wl, L, pg)
    for step in range(steps):
        q, kn, vn = (x.cuda() for x in inputs.step_qkv(wl, layer, step))
        o1, o2 = torch.empty_like(q), torch.empty_like(q)
        sk.decode_step(q, kn, vn, L.k, L.v, L.cache_off, L.len, o1, ws, wl.w, layer, wl.l0)
        sk.decode_step_paged(q, kn, vn, pg.k, pg.v, pg.table, pg.len, o2, ws2, wl.w, layer, wl.l0)
        H.assert_close(H.f64(o2), H.f64(o1), "bf16", f"step {step}")
    assert sk.check_device_error() == sk.OK
    _same_cache(wl, L, pg)


def test_paged_matches_oracle(oracle):
    """Qwen3 shapes, one 30 s request, pooled layer, block size 32: the paged
    fused steps against the oracle's pooling, appends and attention."""
    sk = H.lib()
    wl = inputs.qwen_single()
    layer, steps = wl.l0, 3
    L, pg, (ks, vs, gate) = _prefill_both(wl, layer, steps, 32, seed=5)
    oc = H.oracle_prefill(oracle, wl, layer, steps, ks, vs, gate)
    ws = sk.new_workspace(wl.B, wl.H_q, wl.H_kv, wl.d)
    for step in range(steps):
        q, kn, vn = inputs.step_qkv(wl, layer, step)
        out = torch.empty_like(q, device="cuda")
        sk.decode_step_paged(q.cuda(), kn.cuda(), vn.cuda(), pg.k, pg.v, pg.table, pg.len, out,
                             ws, wl.w, layer, wl.l0)
        ref = []
        for b in range(wl.B):
            Kc, Vc, n = oc[b]
            n = oracle.append_request(Kc, Vc, n, H.f64(kn[b]), H.f64(vn[b]))
            oc[b][2] = n
            ref.append(oracle.decode_attn_request(H.f64(q[b]), Kc[:n], Vc[:n],
                                                  storage=oracle.STORE_BF16))
        H.assert_close(H.f64(out), np.stack(ref), "bf16", f"step {step}")
    assert sk.check_device_error() == sk.OK


def test_paged_tiny_fp32():
    """The tiny fp32 workload (d = 64, 16 text rows + 16 pooled rows), block
    size 8."""
    sk = H.lib()
    wl = inputs.tiny_fp32()
    L, pg, _ = _prefill_both(wl, 0, 4, 8, seed=9)
    _same_cache(wl, L, pg)
    ws = sk.new_workspace(wl.B, wl.H_q, wl.H_kv, wl.d)
    ws2 = sk.new_workspace(wl.B, wl.H_q, wl.H_kv, wl.d)
    for step in range(4):
        q, kn, vn = (x.cuda() for x in inputs.step_qkv(wl, 0, step))
        o1, o2 = torch.empty_like(q), torch.empty_like(q)
        sk.decode_step(q, kn, vn, L.k, L.v, L.cache_off, L.len, o1, ws, wl.w, 0, wl.l0)
        sk.decode_step_paged(q, kn, vn, pg.k, pg.v, pg.table, pg.len, o2, ws2, wl.w, 0, wl.l0)
        assert torch.equal(o1, o2)
    assert sk.check_device_error() == sk.OK


def test_paged_invalid_block_is_reported():
    """A block-table entry of -1 where the next token must go: the append
    reports an invalid argument and writes nothing (no fault)."""
    sk = H.lib()
    wl = inputs.qwen_ragged(B=3)
    wl = dataclasses.replace(wl, G=[0] * wl.B)
    layer = wl.l0
    L, pg, _ = _prefill_both(wl, layer, 64, 64, seed=11)
    table = pg.table.clone()
    n0 = int(pg.len[0])
    table[0, n0 // 64] = -1
    before = pg.k.clone()
    kn = torch.ones((wl.B, wl.H_kv, wl.d), dtype=torch.bfloat16, device="cuda")
    sk.append_paged(kn, kn, pg.k, pg.v, table, pg.len, wl.w, layer, wl.l0)
    assert sk.check_device_error() == sk.ERR_INVALID_ARG
    assert int(pg.len[0]) == n0            # request 0 untouched
    assert int(pg.len[1]) == int(L.len[1]) + 1
    changed = (pg.k != before).any(dim=(1, 2, 3)).nonzero().flatten().tolist()
    tb = pg.table.cpu().numpy()
    for b in (1, 2):                        # only the other requests' pages changed
        n = int(L.len[b])
        assert int(tb[b, n // 64]) in changed
    assert all(int(x) in {int(tb[1, int(L.len[1]) // 64]), int(tb[2, int(L.len[2]) // 64])}
               for x in changed)


def _prefill_q(wl, layer):
    qs = [inputs.prefill_q(wl, layer, b) for b in range(wl.B)]
    q_off = torch.from_numpy(np.concatenate([[0], np.cumsum(wl.full_rows())]).astype(np.int64))
    return torch.cat(qs).cuda(), q_off.cuda()


@pytest.mark.parametrize("block_size,layer", [(8, 8), (16, 8), (64, 8), (128, 8), (256, 8),
                                              (16, 0), (128, 0)])
def test_paged_prefill_matches_contiguous(block_size, layer):
    """speechkv_prefill_attn_paged over the pages speechkv_pool_paged wrote:
    bit-identical to speechkv_prefill_attn over the contiguous cache (a
    pooled layer and a full-resolution one; pages smaller than, equal to and
    larger than a 128-row key tile)."""
    sk = H.lib()
    wl = inputs.qwen_ragged(B=4)
    wl = dataclasses.replace(wl, G=[0] * wl.B)  # the prompt only (before any decoding)
    L, pg, _ = _prefill_both(wl, layer, 0, block_size, seed=block_size + layer)
    _same_cache(wl, L, pg)
    q, q_off = _prefill_q(wl, layer)
    P, T, N = H.lengths_dev(wl)
    o1, o2 = torch.full_like(q, 7.0), torch.full_like(q, 5.0)
    sk.prefill_attn(q, q_off, P, T, N, L.k, L.v, L.cache_off, o1, wl.w, layer, wl.l0, wl.H_kv)
    sk.prefill_attn_paged(q, q_off, P, T, N, pg.k, pg.v, pg.table, o2, wl.w, layer, wl.l0)
    assert sk.check_device_error() == sk.OK
    assert torch.equal(o1, o2)


def test_paged_prefill_invalid_block_is_reported():
    """A block-table entry of -1 inside a request's rows: the paged prefill
    reports an invalid argument (the rows are read from page 0 instead, no
    fault); the other requests' outputs are unaffected."""
    sk = H.lib()
    wl = inputs.qwen_ragged(B=3)
    wl = dataclasses.replace(wl, G=[0] * wl.B)
    layer = wl.l0
    L, pg, _ = _prefill_both(wl, layer, 0, 16, seed=12)
    table = pg.table.clone()
    table[0, 1] = -1
    q, q_off = _prefill_q(wl, layer)
    P, T, N = H.lengths_dev(wl)
    o1, o2 = torch.zeros_like(q), torch.zeros_like(q)
    sk.prefill_attn(q, q_off, P, T, N, L.k, L.v, L.cache_off, o1, wl.w, layer, wl.l0, wl.H_kv)
    assert sk.check_device_error() == sk.OK
    sk.prefill_attn_paged(q, q_off, P, T, N, pg.k, pg.v, table, o2, wl.w, layer, wl.l0)
    assert sk.check_device_error() == sk.ERR_INVALID_ARG
    off = q_off.cpu().numpy()
    assert torch.equal(o1[off[1]:], o2[off[1]:])
