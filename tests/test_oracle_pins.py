"""Pins of the CPU oracle against facts fixed outside the oracle itself.

Each test checks the oracle against a closed form, an invariant the paper's
definitions imply, a library routine, or an independently written brute
force -- never against a retyped copy of the oracle's own formula.

Paper passages (Sec. III-B "SpeechKV"): Eq. (pool) defines the window
softmax gate and the pooled key/value; Eq. (attn) defines the attention of
full-resolution queries over the compressed cache; the gate starts at zero,
i.e. uniform averaging; text positions are left unchanged; layers from l0 on
are pooled.  Sec. V-D gives the 2.8x / 4x cache reductions.
"""
import math
import os

import numpy as np
import pytest
import scipy.special
import torch

from paper_2607_06827_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rand(seed, *shape):
    return np.random.default_rng(seed).standard_normal(shape)


def _to_storage(x, storage):
    """Library rounding of exact values to a storage type: numpy's float32
    conversion (IEEE round to nearest even); torch's bf16 of that fp32 value
    (equal to bf16 of the exact value except at double-rounding ties, which
    random data does not hit)."""
    f32 = np.asarray(x, dtype=np.float64).astype(np.float32)
    if storage == 1:
        return f32.astype(np.float64)
    return torch.from_numpy(f32).to(torch.bfloat16).double().numpy()


def _read_golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            rows.append(dict(kv.split("=") for kv in line.split()))
    return rows


# --------------------------------------------------------------------------
# storage rounding
# --------------------------------------------------------------------------
def test_round_bf16_matches_torch_on_fp32_values(oracle):
    x = np.random.default_rng(0).standard_normal(20000).astype(np.float32)
    x = np.concatenate([x * 1e-3, x, x * 1e3,
                        np.float32([1 + 2**-8, 1 + 3 * 2**-8, -(1 + 2**-8),
                                    2**-134, 3 * 2**-134, 1e-39, 3e38, 0.0])])
    ref = torch.from_numpy(x).to(torch.bfloat16).double().numpy()
    got = np.array([oracle.round_bf16(float(v)) for v in x])
    np.testing.assert_array_equal(got, ref)


def test_round_bf16_ties_to_even(oracle):
    assert oracle.round_bf16(1 + 2**-8) == 1.0            # tie, 1.0 is even
    assert oracle.round_bf16(1 + 3 * 2**-8) == 1 + 2**-6  # tie, rounds up
    assert oracle.round_bf16(1 + 2**-8 + 2**-30) == 1 + 2**-7
    assert math.isinf(oracle.round_bf16(3.5e38))


def test_round_f32_is_ieee_single(oracle):
    x = _rand(1, 1000)
    np.testing.assert_array_equal(
        [oracle.round_f32(v) for v in x], x.astype(np.float32).astype(np.float64))


# --------------------------------------------------------------------------
# length bookkeeping
# --------------------------------------------------------------------------
def test_compressed_len_brute_force(oracle):
    for T in range(0, 40):
        for w in range(1, 10):
            for layer, l0 in ((0, 0), (3, 5), (5, 5), (7, 2)):
                we = w if layer >= l0 else 1
                n = math.ceil(T / we)
                for P, N, G in ((0, 0, 0), (16, 0, 3), (2, 32, 0)):
                    assert oracle.compressed_len(P, T, N, G, w, layer, l0) == P + n + N + G


def test_compressed_len_workload_values(oracle):
    # 30 s of audio at 80 ms/frame pooled with w=4 -> 94 entries (+32 prompt).
    T = inputs.frames_from_seconds(30)
    assert T == 375
    assert oracle.compressed_len(0, T, 32, 0, 4, 8, 8) == 94 + 32
    assert oracle.compressed_len(0, T, 32, 0, 4, 7, 8) == 375 + 32
    # tiny case: 16 text + 64 frames / 4, then 8 appended tokens
    assert [oracle.compressed_len(16, 64, 0, g, 4, 0, 0) for g in range(1, 9)] == list(range(33, 41))
    assert [oracle.compressed_len(16, 64, 0, g, 1, 0, 0) for g in range(1, 9)] == list(range(81, 89))
    assert oracle.compressed_len(0, 0, 0, 0, 4, 9, 0) == 0
    assert oracle.compressed_len(0, 3, 0, 0, 4, 9, 0) == 1          # T < w
    assert oracle.compressed_len(-1, 3, 0, 0, 4, 9, 0) == -1         # bad args
    assert oracle.compressed_len(0, 3, 0, 0, 0, 9, 0) == -1


def test_memory_reduction_matches_paper(oracle):
    """Sec. V-D: the speech cache shrinks 2.8x at R=4 and 4x at R=8 with the
    paper's l0 = 5 (1-indexed: first 4 of 28 layers uncompressed)."""
    for row in _read_golden("memory_reduction.txt"):
        R, layers = int(row["R"]), int(row["layers"])
        l0 = int(row["l0_paper"]) - 1          # paper counts layers from 1
        T = 15000                              # speech only, T divisible by R
        full = sum(oracle.compressed_len(0, T, 0, 0, 1, l, 0) for l in range(layers))
        comp = sum(oracle.compressed_len(0, T, 0, 0, R, l, l0) for l in range(layers))
        assert full / comp == pytest.approx(float(row["reduction"]), abs=1e-12)


# --------------------------------------------------------------------------
# pooling, Eq. (pool)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("w,layer,l0", [(1, 3, 0), (4, 2, 3), (8, 0, 1)])
def test_pool_identity_when_not_pooled(oracle, w, layer, l0):
    """w_eff = 1 (w = 1, or a layer before l0): alpha = 1 exactly, so the
    cache is a bit-exact copy of the prefill rows."""
    P, T, N, H, d = 3, 11, 5, 2, 8
    K, V = _rand(2, P + T + N, H, d), _rand(3, P + T + N, H, d)
    Ko, Vo = oracle.pool_request(K, V, P, T, N, _rand(4, H, d), w, layer, l0)
    np.testing.assert_array_equal(Ko, K)
    np.testing.assert_array_equal(Vo, V)


@pytest.mark.parametrize("P,T,N,w", [(16, 64, 0, 4), (0, 375, 32, 4),
                                     (2, 10, 3, 3), (0, 3, 1, 4), (1, 0, 2, 4),
                                     (0, 13, 0, 8)])
def test_pool_zero_gate_is_window_mean(oracle, P, T, N, w):
    """Zero gate (the paper's initialisation): uniform weights, i.e. the plain
    mean of each window; the short last window averages what it holds; text
    rows keep their place before and after the pooled speech."""
    H, d = 2, 8
    K, V = _rand(5, P + T + N, H, d), _rand(6, P + T + N, H, d)
    Ko, Vo = oracle.pool_request(K, V, P, T, N, np.zeros((H, d)), w, 1, 0)
    n = -(-T // w)
    assert Ko.shape == (P + n + N, H, d)
    np.testing.assert_array_equal(Ko[:P], K[:P])
    np.testing.assert_array_equal(Ko[P + n:], K[P + T:])
    for i in range(n):
        sl = slice(P + i * w, P + min((i + 1) * w, T))
        np.testing.assert_allclose(Ko[P + i], K[sl].mean(axis=0), rtol=0, atol=1e-14)
        np.testing.assert_allclose(Vo[P + i], V[sl].mean(axis=0), rtol=0, atol=1e-14)


def test_pool_two_frame_window_is_logistic(oracle):
    """With two frames, alpha_1 = 1 / (1 + exp(z_2 - z_1)) (logistic)."""
    H, d = 3, 16
    K, V = _rand(7, 2, H, d), _rand(8, 2, H, d)
    u = _rand(9, H, d)
    Ko, Vo, alpha = oracle.pool_request(K, V, 0, 2, 0, u, 2, 0, 0, want_alpha=True)
    for h in range(H):
        z = K[:, h] @ u[h]
        a1 = scipy.special.expit(z[0] - z[1])
        assert alpha[0, h] == pytest.approx(a1, rel=1e-13)
        np.testing.assert_allclose(Ko[0, h], a1 * K[0, h] + (1 - a1) * K[1, h], atol=1e-13)
        np.testing.assert_allclose(Vo[0, h], a1 * V[0, h] + (1 - a1) * V[1, h], atol=1e-13)


def test_pool_brute_force(oracle):
    """Independent restatement: per window exp(z)/sum(exp(z)) with no max
    subtraction, weights from the keys applied to keys and values."""
    P, T, N, H, d, w = 4, 37, 6, 3, 16, 5
    K, V = _rand(10, P + T + N, H, d), _rand(11, P + T + N, H, d)
    u = _rand(12, H, d) / 4
    Ko, Vo = oracle.pool_request(K, V, P, T, N, u, w, 2, 2)
    rows_k, rows_v = list(K[:P]), list(V[:P])
    for start in range(P, P + T, w):
        fr = range(start, min(start + w, P + T))
        kk = np.zeros((H, d)); vv = np.zeros((H, d))
        for h in range(H):
            ex = [math.exp(sum(u[h, c] * K[j, h, c] for c in range(d))) for j in fr]
            tot = sum(ex)
            for e, j in zip(ex, fr):
                kk[h] += e / tot * K[j, h]
                vv[h] += e / tot * V[j, h]
        rows_k.append(kk); rows_v.append(vv)
    rows_k += list(K[P + T:]); rows_v += list(V[P + T:])
    np.testing.assert_allclose(Ko, np.array(rows_k), rtol=0, atol=1e-12)
    np.testing.assert_allclose(Vo, np.array(rows_v), rtol=0, atol=1e-12)


def test_pool_dominant_gate_selects_frame_and_drives_values(oracle):
    """A large gate along one coordinate puts all weight on the frame whose key
    is largest there, for the key AND the value (V uses K's weights), and only
    for the head whose gate row is large."""
    H, d, w, T = 2, 8, 4, 8
    K, V = _rand(13, T, H, d), _rand(14, T, H, d)
    u = np.zeros((H, d)); u[1, 0] = 1e4
    Ko, Vo = oracle.pool_request(K, V, 0, T, 0, u, w, 0, 0)
    for i in range(T // w):
        win = slice(i * w, (i + 1) * w)
        jstar = i * w + int(np.argmax(K[win, 1, 0]))
        np.testing.assert_allclose(Ko[i, 1], K[jstar, 1], atol=1e-12)
        np.testing.assert_allclose(Vo[i, 1], V[jstar, 1], atol=1e-12)
        np.testing.assert_allclose(Ko[i, 0], K[win, 0].mean(axis=0), atol=1e-14)


def test_pool_invariances(oracle):
    P, T, N, H, d, w = 0, 24, 0, 2, 8, 4
    K, V = _rand(15, T, H, d), _rand(16, T, H, d)
    u = _rand(17, H, d)
    Ko, Vo, alpha = oracle.pool_request(K, V, P, T, N, u, w, 0, 0, want_alpha=True)
    # weights of a window sum to one and are positive
    np.testing.assert_allclose(alpha.reshape(T // w, w, H).sum(axis=1), 1.0, atol=1e-14)
    assert (alpha > 0).all()
    # order of frames inside a window does not matter ...
    perm = np.concatenate([i * w + np.random.default_rng(i).permutation(w)
                           for i in range(T // w)])
    Kp, Vp = oracle.pool_request(K[perm], V[perm], P, T, N, u, w, 0, 0)
    np.testing.assert_allclose(Kp, Ko, atol=1e-13)
    np.testing.assert_allclose(Vp, Vo, atol=1e-13)
    # ... but moving frames across windows does
    Kx, _ = oracle.pool_request(K[::-1].copy(), V[::-1].copy(), P, T, N, u, w, 0, 0)
    assert np.abs(Kx - Ko).max() > 1e-3
    # a common shift delta of every key in a window shifts every logit by u.delta,
    # leaving alpha alone: K-hat moves by delta, V-hat does not move
    delta = _rand(18, H, d)
    Ks, Vs = oracle.pool_request(K + delta[None], V, P, T, N, u, w, 0, 0)
    np.testing.assert_allclose(Ks, Ko + delta[None], atol=1e-12)
    np.testing.assert_allclose(Vs, Vo, atol=1e-12)
    # values equal to keys pool to the pooled keys; constant values stay put
    Kk, Vk = oracle.pool_request(K, K, P, T, N, u, w, 0, 0)
    np.testing.assert_array_equal(Vk, Kk)
    c = _rand(19, H, d)
    _, Vc = oracle.pool_request(K, np.broadcast_to(c, (T, H, d)), P, T, N, u, w, 0, 0)
    np.testing.assert_allclose(Vc, np.broadcast_to(c, Vc.shape), atol=1e-14)


def test_pool_storage_rounding(oracle):
    H, d = 2, 8
    K, V = _rand(20, 8, H, d), _rand(21, 8, H, d)
    u = _rand(22, H, d)
    Ke, Ve = oracle.pool_request(K, V, 0, 8, 0, u, 4, 0, 0)
    Kb, Vb = oracle.pool_request(K, V, 0, 8, 0, u, 4, 0, 0, storage=oracle.STORE_BF16)
    ref = torch.from_numpy(Ke).float().to(torch.bfloat16).double().numpy()
    # bf16 of the exact value; equal to torch's bf16 of the fp32 value except
    # at double-rounding ties, which random data does not hit
    np.testing.assert_array_equal(Kb, ref)
    assert np.abs(Kb - Ke).max() <= 2**-8 * np.abs(Ke).max()


def test_pool_text_rows_rounded_once(oracle):
    """Text rows (before and after the speech) are copied and rounded once to
    the storage type, like every other value the pooling produces."""
    P, T, N, H, d, w = 3, 8, 2, 2, 8, 4
    K, V = _rand(23, P + T + N, H, d), _rand(24, P + T + N, H, d)
    u = _rand(25, H, d)
    n = -(-T // w)
    for storage in (oracle.STORE_F32, oracle.STORE_BF16):
        Ko, Vo = oracle.pool_request(K, V, P, T, N, u, w, 0, 0, storage=storage)
        for src, out in ((K, Ko), (V, Vo)):
            text_in = np.concatenate([src[:P], src[P + T:]])
            text_out = np.concatenate([out[:P], out[P + n:]])
            assert not np.array_equal(text_out, text_in)
            np.testing.assert_array_equal(text_out, _to_storage(text_in, storage))


# --------------------------------------------------------------------------
# append
# --------------------------------------------------------------------------
def test_append_places_row_and_respects_capacity(oracle):
    H, d, cap = 2, 4, 3
    Kc = np.zeros((cap, H, d)); Vc = np.zeros((cap, H, d))
    n = 0
    for t in range(cap):
        k, v = np.full((H, d), t + 1.0), np.full((H, d), -(t + 1.0))
        n = oracle.append_request(Kc, Vc, n, k, v)
        assert n == t + 1
        np.testing.assert_array_equal(Kc[t], k)
        np.testing.assert_array_equal(Vc[t], v)
    before = Kc.copy()
    assert oracle.append_request(Kc, Vc, n, np.ones((H, d)), np.ones((H, d))) == -1
    np.testing.assert_array_equal(Kc, before)


# --------------------------------------------------------------------------
# decode attention, Eq. (attn)
# --------------------------------------------------------------------------
def _sdpa_gqa(q, K, V, scale=None):
    """torch CPU fp64 scaled_dot_product_attention with KV heads repeated."""
    H_q, d = q.shape
    n, H_kv, _ = K.shape
    G = H_q // H_kv
    qt = torch.from_numpy(q)[:, None, :]                                # [H_q,1,d]
    kt = torch.from_numpy(K).permute(1, 0, 2).repeat_interleave(G, 0)  # [H_q,n,d]
    vt = torch.from_numpy(V).permute(1, 0, 2).repeat_interleave(G, 0)
    o = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, scale=scale)
    return o[:, 0, :].numpy()


@pytest.mark.parametrize("H_q,H_kv,d,n", [(4, 2, 64, 40), (16, 8, 128, 126),
                                          (6, 3, 16, 1), (8, 1, 32, 300)])
def test_attn_matches_sdpa(oracle, H_q, H_kv, d, n):
    q, K, V = _rand(30, H_q, d), _rand(31, n, H_kv, d), _rand(32, n, H_kv, d)
    np.testing.assert_allclose(oracle.decode_attn_request(q, K, V),
                               _sdpa_gqa(q, K, V), rtol=0, atol=1e-12)
    np.testing.assert_allclose(oracle.decode_attn_request(q, K, V, scale=0.3),
                               _sdpa_gqa(q, K, V, scale=0.3), rtol=0, atol=1e-12)


def test_attn_brute_force_tiny_case(oracle):
    """The tiny fp32 workload's shapes; explicit triple loop, no max
    subtraction, exp/sum straight from the softmax definition."""
    wl = inputs.tiny_fp32()
    H_q, H_kv, d, n = wl.H_q, wl.H_kv, wl.d, 40
    q, K, V = _rand(33, H_q, d), _rand(34, n, H_kv, d), _rand(35, n, H_kv, d)
    out = oracle.decode_attn_request(q, K, V)
    G = H_q // H_kv
    ref = np.zeros((H_q, d))
    for hq in range(H_q):
        h = hq // G
        e = [math.exp(sum(q[hq, c] * K[j, h, c] for c in range(d)) / math.sqrt(d))
             for j in range(n)]
        tot = sum(e)
        for c in range(d):
            ref[hq, c] = sum(e[j] / tot * V[j, h, c] for j in range(n))
    np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)


def test_attn_invariants(oracle):
    H_q, H_kv, d, n = 4, 2, 16, 23
    q, K, V = _rand(36, H_q, d), _rand(37, n, H_kv, d), _rand(38, n, H_kv, d)
    _, probs = oracle.decode_attn_request(q, K, V, want_probs=True)
    np.testing.assert_allclose(probs.sum(axis=1), 1.0, atol=1e-14)
    assert (probs >= 0).all()
    # equal keys or a zero query: plain mean of the values of the group's head
    Ke = np.broadcast_to(K[:1], K.shape).copy()
    G = H_q // H_kv
    for out in (oracle.decode_attn_request(q, Ke, V),
                oracle.decode_attn_request(np.zeros_like(q), K, V)):
        for hq in range(H_q):
            np.testing.assert_allclose(out[hq], V[:, hq // G].mean(axis=0), atol=1e-14)
    # a single cached entry returns its value
    out1 = oracle.decode_attn_request(q, K[:1], V[:1])
    for hq in range(H_q):
        np.testing.assert_allclose(out1[hq], V[0, hq // G], atol=0)
    # empty cache: zeros by convention
    assert not oracle.decode_attn_request(q, K[:0], V[:0]).any()
    # scale 0 means 1/sqrt(d)
    np.testing.assert_array_equal(oracle.decode_attn_request(q, K, V, scale=0.0),
                                  oracle.decode_attn_request(q, K, V, scale=1 / math.sqrt(d)))


def test_attn_gqa_head_mapping(oracle):
    """Query heads 0..G-1 read KV head 0, heads G..2G-1 read KV head 1."""
    H_q, H_kv, d, n = 4, 2, 8, 5
    K = _rand(39, n, H_kv, d)
    V = np.zeros((n, H_kv, d)); V[:, 0] = 1.0; V[:, 1] = 2.0
    out = oracle.decode_attn_request(_rand(40, H_q, d), K, V)
    np.testing.assert_allclose(out[:2], 1.0, atol=1e-14)
    np.testing.assert_allclose(out[2:], 2.0, atol=1e-14)


def test_attn_extreme_logits(oracle):
    """A huge query scale gives a finite result equal to the value of the
    best-scoring key (softmax becomes one-hot)."""
    H_q, H_kv, d, n = 2, 1, 16, 50
    q, K, V = _rand(41, H_q, d) * 1e4, _rand(42, n, H_kv, d), _rand(43, n, H_kv, d)
    for shift in range(n):          # put the best key at every position
        Ks, Vs = np.roll(K, shift, axis=0), np.roll(V, shift, axis=0)
        out = oracle.decode_attn_request(q, Ks, Vs)
        assert np.isfinite(out).all()
        for hq in range(H_q):
            best = int(np.argmax(Ks[:, 0] @ q[hq]))
            np.testing.assert_allclose(out[hq], Vs[best, 0], atol=1e-12)


def test_attn_output_rounded_once(oracle):
    """The attention output is the exact result rounded once to storage."""
    H_q, H_kv, d, n = 4, 2, 16, 33
    q, K, V = _rand(44, H_q, d), _rand(45, n, H_kv, d), _rand(46, n, H_kv, d)
    exact = oracle.decode_attn_request(q, K, V)
    for storage in (oracle.STORE_F32, oracle.STORE_BF16):
        out = oracle.decode_attn_request(q, K, V, storage=storage)
        assert not np.array_equal(out, exact)
        np.testing.assert_array_equal(out, _to_storage(exact, storage))


# --------------------------------------------------------------------------
# whole step: w = 1 is plain uncompressed attention
# --------------------------------------------------------------------------
def test_w1_pipeline_is_uncompressed_attention(oracle):
    """The MLP baseline (no pooling) equals SpeechKV with w = 1: pooling,
    appending decoded tokens and attending must reproduce plain attention over
    the full-resolution sequence."""
    P, T, N, H_q, H_kv, d, steps = 5, 30, 7, 4, 2, 16, 4
    S = P + T + N
    K, V = _rand(50, S, H_kv, d), _rand(51, S, H_kv, d)
    Ko, Vo = oracle.pool_request(K, V, P, T, N, _rand(52, H_kv, d), 1, 0, 0)
    Kc = np.zeros((S + steps, H_kv, d)); Vc = np.zeros_like(Kc)
    Kc[:S], Vc[:S] = Ko, Vo
    n = S
    Kfull, Vfull = K.copy(), V.copy()
    for t in range(steps):
        kn, vn, q = _rand(60 + t, H_kv, d), _rand(70 + t, H_kv, d), _rand(80 + t, H_q, d)
        n = oracle.append_request(Kc, Vc, n, kn, vn)
        Kfull = np.concatenate([Kfull, kn[None]]); Vfull = np.concatenate([Vfull, vn[None]])
        np.testing.assert_allclose(oracle.decode_attn_request(q, Kc[:n], Vc[:n]),
                                   _sdpa_gqa(q, Kfull, Vfull), rtol=0, atol=1e-12)


# --------------------------------------------------------------------------
# prefill attention (Eq. (attn) with the adjusted causal mask)
# --------------------------------------------------------------------------
def _first_source(P, T, N, w):
    """Prompt position of the first frame behind each compressed row: the
    text prefix maps to itself, pooled window i starts at frame P + i*w, the
    text after the speech sits T - n positions further on.  Written from the
    row order of the compressed cache, not from the oracle."""
    n = -(-T // w)
    return [e for e in range(P)] + [P + i * w for i in range(n)] + \
        [P + T + j for j in range(N)]


def _visible(P, T, N, w):
    """mask[t][e]: compressed row e precedes prompt position t (its first
    source frame is not after t)."""
    src = np.array(_first_source(P, T, N, w))
    t = np.arange(P + T + N)
    return src[None, :] <= t[:, None]


@pytest.mark.parametrize("P,T,N,w", [(0, 375, 32, 4), (16, 64, 0, 4), (3, 10, 5, 3),
                                     (2, 7, 3, 8), (0, 1, 1, 4), (5, 0, 4, 4), (4, 9, 2, 1)])
def test_prefill_position_is_last_visible_row(oracle, P, T, N, w):
    mask = _visible(P, T, N, w)
    for t in range(P + T + N):
        vis = np.nonzero(mask[t])[0]
        # the visible rows are a prefix, and pi(t) is its last row
        assert list(vis) == list(range(len(vis)))
        assert oracle.prefill_position(P, T, N, w, t) == vis[-1]
    assert oracle.prefill_position(P, T, N, w, P + T + N - 1) == mask.shape[1] - 1


def _sdpa_causal(Q, K, V, mask=None):
    """torch scaled_dot_product_attention in fp64, GQA by repeating KV heads."""
    G = Q.shape[1] // K.shape[1]
    qt = torch.from_numpy(Q).permute(1, 0, 2)
    kt = torch.from_numpy(K).permute(1, 0, 2).repeat_interleave(G, 0)
    vt = torch.from_numpy(V).permute(1, 0, 2).repeat_interleave(G, 0)
    if mask is None:
        o = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True)
    else:
        o = torch.nn.functional.scaled_dot_product_attention(
            qt, kt, vt, attn_mask=torch.from_numpy(mask))
    return o.permute(1, 0, 2).numpy()


@pytest.mark.parametrize("P,T,N,H_q,H_kv,d", [(4, 30, 6, 4, 2, 16), (0, 50, 0, 2, 2, 8),
                                              (7, 0, 3, 6, 3, 32)])
def test_prefill_w1_is_causal_attention(oracle, P, T, N, H_q, H_kv, d):
    """Without pooling the prefill is plain causal attention (the library's)."""
    S = P + T + N
    Q, K, V = _rand(90, S, H_q, d), _rand(91, S, H_kv, d), _rand(92, S, H_kv, d)
    np.testing.assert_allclose(oracle.prefill_attn_request(Q, K, V, P, T, N, 1),
                               _sdpa_causal(Q, K, V), rtol=0, atol=1e-12)


@pytest.mark.parametrize("P,T,N,w", [(0, 37, 8, 4), (5, 20, 3, 3), (2, 7, 0, 8)])
def test_prefill_matches_masked_sdpa(oracle, P, T, N, w):
    """Pooled layer: the library's attention with the mask of the window
    sources gives the same rows."""
    H_q, H_kv, d = 4, 2, 16
    c = len(_first_source(P, T, N, w))
    Q, K, V = _rand(93, P + T + N, H_q, d), _rand(94, c, H_kv, d), _rand(95, c, H_kv, d)
    np.testing.assert_allclose(oracle.prefill_attn_request(Q, K, V, P, T, N, w),
                               _sdpa_causal(Q, K, V, _visible(P, T, N, w)), rtol=0, atol=1e-12)


def test_prefill_last_row_is_decode_attention(oracle):
    """The last prompt position sees the whole compressed cache: its row is
    the decode attention of that query."""
    P, T, N, w, H_q, H_kv, d = 3, 41, 5, 4, 8, 4, 32
    c = len(_first_source(P, T, N, w))
    Q, K, V = _rand(96, P + T + N, H_q, d), _rand(97, c, H_kv, d), _rand(98, c, H_kv, d)
    out = oracle.prefill_attn_request(Q, K, V, P, T, N, w)
    np.testing.assert_allclose(out[-1], oracle.decode_attn_request(Q[-1], K, V),
                               rtol=0, atol=1e-12)


def test_prefill_equal_keys_average_visible_values(oracle):
    """All keys of a head equal: the softmax is uniform, so each query gets
    the running mean of the values it may see."""
    P, T, N, w, H_q, H_kv, d = 2, 13, 3, 4, 4, 2, 8
    mask = _visible(P, T, N, w)
    c = mask.shape[1]
    Q, V = _rand(99, P + T + N, H_q, d), _rand(100, c, H_kv, d)
    K = np.repeat(_rand(101, 1, H_kv, d), c, axis=0)
    out = oracle.prefill_attn_request(Q, K, V, P, T, N, w)
    for t in range(P + T + N):
        for hq in range(H_q):
            ref = V[mask[t], hq // 2].mean(axis=0)
            np.testing.assert_allclose(out[t, hq], ref, rtol=0, atol=1e-12)


def test_prefill_output_rounded_once(oracle):
    """Each prefill output row is the exact result rounded once to storage."""
    P, T, N, w, H_q, H_kv, d = 2, 11, 3, 4, 4, 2, 16
    c = len(_first_source(P, T, N, w))
    Q, K, V = _rand(102, P + T + N, H_q, d), _rand(103, c, H_kv, d), _rand(104, c, H_kv, d)
    exact = oracle.prefill_attn_request(Q, K, V, P, T, N, w)
    for storage in (oracle.STORE_F32, oracle.STORE_BF16):
        out = oracle.prefill_attn_request(Q, K, V, P, T, N, w, storage=storage)
        assert not np.array_equal(out, exact)
        np.testing.assert_array_equal(out, _to_storage(exact, storage))


def test_prefill_brute_force_tiny_case(oracle):
    """Explicit loops from the definitions: mask from the window sources,
    exp without max subtraction, scale 1/sqrt(d)."""
    P, T, N, w, H_q, H_kv, d = 2, 7, 3, 3, 4, 2, 8
    mask = _visible(P, T, N, w)
    c = mask.shape[1]
    Q, K, V = _rand(102, P + T + N, H_q, d), _rand(103, c, H_kv, d), _rand(104, c, H_kv, d)
    out = oracle.prefill_attn_request(Q, K, V, P, T, N, w)
    for t in range(P + T + N):
        for hq in range(H_q):
            h = hq // (H_q // H_kv)
            e = [math.exp(sum(Q[t, hq, k] * K[j, h, k] for k in range(d)) / math.sqrt(d))
                 if mask[t, j] else 0.0 for j in range(c)]
            tot = sum(e)
            for k in range(d):
                ref = sum(e[j] / tot * V[j, h, k] for j in range(c))
                assert abs(out[t, hq, k] - ref) < 1e-12
