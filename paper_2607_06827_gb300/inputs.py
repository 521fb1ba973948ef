"""Seeded synthetic inputs for SpeechKV workloads.

This module draws lengths and tensors only; it holds none of the method's
arithmetic (no pooling, no window counts, no attention).  Both the CUDA path's
tests/bench and the CPU oracle's tests take their inputs from here.

Shapes follow the paper's setting (Sec. IV-A): a Qwen3-1.7B backbone (28
decoder layers, 16 query heads, 8 KV heads, head dim 128) fed one speech frame
per 80 ms.  Values: Q/K/V ~ N(0, 1); gate vectors u ~ N(0, 1/d) so that a gate
logit u.k has unit variance on unit-variance keys.  CPU tensors come from
numpy's PCG64 (fp32 draws, rounded to bf16 where bf16 storage applies); large
benchmark tensors are drawn on the device with torch's Philox generator.
"""
from __future__ import annotations

import dataclasses
from typing import List

import numpy as np

FRAME_MS = 80          # one speech frame per 80 ms (Sec. IV-A)
QWEN3_1P7B = dict(L=28, H_q=16, H_kv=8, d=128)


def frames_from_seconds(sec: float) -> int:
    """Number of 80 ms frames covering ``sec`` seconds (rounded up)."""
    ms = int(round(sec * 1000))
    return (ms + FRAME_MS - 1) // FRAME_MS


@dataclasses.dataclass
class Workload:
    """One synthetic decode workload.

    Per request b: P[b] text tokens before the speech, T[b] speech frames,
    N[b] text tokens after the speech, G[b] tokens already generated before
    the first timed/checked step.  ``steps`` decode steps follow.
    """
    name: str
    dtype: str                  # "f32" or "bf16" (storage type)
    L: int                      # layers
    l0: int                     # first pooled layer (0-indexed)
    w: int                      # pooling window
    H_q: int
    H_kv: int
    d: int
    P: List[int]
    T: List[int]
    N: List[int]
    G: List[int]
    steps: int
    seed: int

    @property
    def B(self) -> int:
        return len(self.T)

    def full_rows(self) -> List[int]:
        """Prefill rows per request (text + speech + text)."""
        return [p + t + n for p, t, n in zip(self.P, self.T, self.N)]


def tiny_fp32(seed: int = 1001) -> Workload:
    """fp32 correctness case: 1 layer (pooled, l0 = 0), B = 1, 4 query / 2 KV
    heads, d = 64; 16-token text prefix, 64 speech frames, w = 4; 8 steps."""
    return Workload("tiny-fp32", "f32", L=1, l0=0, w=4, H_q=4, H_kv=2, d=64,
                    P=[16], T=[64], N=[0], G=[0], steps=8, seed=seed)


def qwen_single(seed: int = 1002, layers: int | None = None) -> Workload:
    """Qwen3-1.7B shapes, bf16, B = 1: 30 s audio (375 frames), w = 4, 32-token
    prompt after the speech, l0 = 8, 128 decode steps."""
    s = QWEN3_1P7B
    return Workload("qwen-b1-30s", "bf16", L=layers or s["L"], l0=8, w=4,
                    H_q=s["H_q"], H_kv=s["H_kv"], d=s["d"], P=[0],
                    T=[frames_from_seconds(30)], N=[32], G=[0], steps=128,
                    seed=seed)


def qwen_batch64(w: int = 4, seed: int = 1003) -> Workload:
    """Qwen3-1.7B shapes, bf16, 64 uniform requests of 30 s audio, 32-token
    prompt, 256 decode steps; the w = 1 twin uses the same seed."""
    s = QWEN3_1P7B
    B = 64
    return Workload(f"qwen-b64-30s-w{w}", "bf16", L=s["L"], l0=8, w=w,
                    H_q=s["H_q"], H_kv=s["H_kv"], d=s["d"], P=[0] * B,
                    T=[frames_from_seconds(30)] * B, N=[32] * B, G=[0] * B,
                    steps=256, seed=seed)


LONG_AUDIO_MINUTES = (2, 5, 10, 20)


def qwen_long_audio(minutes: int, w: int, seed: int = 1004,
                    generated: int = 0) -> Workload:
    """Qwen3-1.7B shapes, bf16, B = 8: ``minutes`` of audio, window w, 64-token
    prompt, l0 = 8, 128 decode steps.  ``generated`` tokens are already in the
    cache before the first step (a mid-run snapshot)."""
    s = QWEN3_1P7B
    B = 8
    T = frames_from_seconds(60 * minutes)
    return Workload(f"qwen-b8-{minutes}min-w{w}", "bf16", L=s["L"], l0=8, w=w,
                    H_q=s["H_q"], H_kv=s["H_kv"], d=s["d"], P=[0] * B,
                    T=[T] * B, N=[64] * B, G=[generated] * B, steps=128,
                    seed=seed)


def qwen_ragged(B: int = 128, w: int = 4, seed: int = 1005) -> Workload:
    """Ragged serving batch at Qwen3-1.7B shapes, bf16: per request audio
    uniform in 5-120 s (63-1500 frames), prompt uniform in 16-256 tokens,
    already-generated tokens uniform in 0-512; all drawn from one seed."""
    s = QWEN3_1P7B
    rng = np.random.default_rng(seed)
    T = rng.integers(frames_from_seconds(5), frames_from_seconds(120),
                     size=B, endpoint=True)
    N = rng.integers(16, 256, size=B, endpoint=True)
    G = rng.integers(0, 512, size=B, endpoint=True)
    return Workload(f"qwen-ragged-b{B}-w{w}", "bf16", L=s["L"], l0=8, w=w,
                    H_q=s["H_q"], H_kv=s["H_kv"], d=s["d"], P=[0] * B,
                    T=[int(x) for x in T], N=[int(x) for x in N],
                    G=[int(x) for x in G], steps=128, seed=seed)


# --------------------------------------------------------------------------
# tensors (CPU, numpy PCG64)
# --------------------------------------------------------------------------
TAG_PREFILL_K, TAG_PREFILL_V, TAG_GATE = 1, 2, 3
TAG_Q, TAG_KNEW, TAG_VNEW, TAG_GEN_K, TAG_GEN_V = 4, 5, 6, 7, 8
TAG_PREFILL_Q = 9
TAG_HIDDEN, TAG_HIDDEN_GATE = 10, 11


def rng_for(seed: int, *key: int) -> np.random.Generator:
    """Independent stream for (seed, key...) via numpy's SeedSequence."""
    return np.random.default_rng(np.random.SeedSequence([seed, *key]))


def normal_f32(seed: int, key, shape, std: float = 1.0) -> np.ndarray:
    """N(0, std^2) fp32 draws from the stream ``rng_for(seed, *key)``."""
    g = rng_for(seed, *key)
    return (g.standard_normal(size=shape, dtype=np.float32)
            * np.float32(std)).astype(np.float32)


def to_storage(x: np.ndarray, dtype: str):
    """fp32 numpy -> torch CPU tensor of the storage dtype (bf16: RNE)."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32))
    return t.to(torch.bfloat16) if dtype == "bf16" else t


def prefill_kv(wl: Workload, layer: int, b: int):
    """Prefill key and value of request b at ``layer``: [P+T+N, H_kv, d]."""
    S = wl.P[b] + wl.T[b] + wl.N[b]
    shape = (S, wl.H_kv, wl.d)
    k = normal_f32(wl.seed, (TAG_PREFILL_K, layer, b), shape)
    v = normal_f32(wl.seed, (TAG_PREFILL_V, layer, b), shape)
    return to_storage(k, wl.dtype), to_storage(v, wl.dtype)


def prefill_q(wl: Workload, layer: int, b: int):
    """Prompt queries of request b at ``layer``: [P+T+N, H_q, d]."""
    S = wl.P[b] + wl.T[b] + wl.N[b]
    q = normal_f32(wl.seed, (TAG_PREFILL_Q, layer, b), (S, wl.H_q, wl.d))
    return to_storage(q, wl.dtype)


def hidden_states(wl: Workload, b: int, d_model: int):
    """Hidden states of request b's prompt at the pooling layer: [P+T+N, d_model]."""
    S = wl.P[b] + wl.T[b] + wl.N[b]
    return to_storage(normal_f32(wl.seed, (TAG_HIDDEN, b), (S, d_model)), wl.dtype)


def hidden_gate(wl: Workload, d_model: int, scale: float = 1.0) -> np.ndarray:
    """Gate vector u ~ N(0, scale^2 / d_model) over the hidden state, fp32 [d_model]."""
    return normal_f32(wl.seed, (TAG_HIDDEN_GATE,), (d_model,), std=scale / np.sqrt(d_model))


def generated_kv(wl: Workload, layer: int, b: int):
    """Keys/values of the G[b] tokens generated before step 0: [G, H_kv, d]."""
    shape = (wl.G[b], wl.H_kv, wl.d)
    k = normal_f32(wl.seed, (TAG_GEN_K, layer, b), shape)
    v = normal_f32(wl.seed, (TAG_GEN_V, layer, b), shape)
    return to_storage(k, wl.dtype), to_storage(v, wl.dtype)


def gate(wl: Workload, layer: int, scale: float = 1.0) -> np.ndarray:
    """Gate vectors u[h] ~ N(0, scale^2 / d), fp32 [H_kv, d]."""
    return normal_f32(wl.seed, (TAG_GATE, layer), (wl.H_kv, wl.d),
                      std=scale / np.sqrt(wl.d))


def step_qkv(wl: Workload, layer: int, step: int):
    """Decode-step inputs at ``layer``: q [B, H_q, d], k_new/v_new [B, H_kv, d]."""
    q = normal_f32(wl.seed, (TAG_Q, layer, step), (wl.B, wl.H_q, wl.d))
    k = normal_f32(wl.seed, (TAG_KNEW, layer, step), (wl.B, wl.H_kv, wl.d))
    v = normal_f32(wl.seed, (TAG_VNEW, layer, step), (wl.B, wl.H_kv, wl.d))
    return (to_storage(q, wl.dtype), to_storage(k, wl.dtype),
            to_storage(v, wl.dtype))


# --------------------------------------------------------------------------
# tensors (device, torch Philox) for benchmark-sized inputs
# --------------------------------------------------------------------------
def device_normal(shape, dtype, device, seed: int, *key: int):
    """N(0, 1) tensor drawn on ``device`` from a generator seeded by
    (seed, key...).  Used where numpy on the host would be too slow."""
    import torch
    mixed = int(np.random.SeedSequence([seed, *key]).generate_state(1)[0])
    g = torch.Generator(device=device)
    g.manual_seed(mixed)
    t = torch.empty(shape, dtype=torch.float32, device=device)
    t.normal_(generator=g)
    return t.to(dtype)
