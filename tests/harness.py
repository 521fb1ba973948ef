"""Test-side plumbing: build the library, lay synthetic workloads out in the
library's cache layout, and turn GPU caches back into per-request arrays for
the oracle.  Holds none of the method's arithmetic: cache capacities come from
the library's own host helper (speechkv_compressed_len) on the GPU side and
from the oracle on the oracle side.
"""
from __future__ import annotations

import os
import sys

import numpy as np
import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2607_06827_gb300 import inputs  # noqa: E402

TORCH_DTYPE = {"f32": torch.float32, "bf16": torch.bfloat16}

# Tolerances: fp32 max-abs 1e-5; bf16 max-abs 2e-2 and mean-abs 2e-3 (unit
# variance inputs).
TOL = {"f32": dict(max_abs=1e-5, mean_abs=1e-5), "bf16": dict(max_abs=2e-2, mean_abs=2e-3)}


def lib():
    from paper_2607_06827_gb300 import build, speechkv
    build.build()
    return speechkv


def require_gpu():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")


def assert_close(got, ref, dtype, what=""):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (what, got.shape, ref.shape)
    assert np.isfinite(got).all(), f"{what}: non-finite values"
    err = np.abs(got - ref)
    tol = TOL[dtype]
    assert err.max() <= tol["max_abs"], f"{what}: max abs err {err.max():.3g} > {tol['max_abs']}"
    assert err.mean() <= tol["mean_abs"], f"{what}: mean abs err {err.mean():.3g} > {tol['mean_abs']}"


def f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().to("cpu", torch.float64).numpy()


class GpuLayer:
    """One layer's packed cache for a workload, in the library's layout."""

    def __init__(self, wl: inputs.Workload, layer: int, extra_rows: int, device="cuda"):
        sk = lib()
        self.wl, self.layer, self.device = wl, layer, device
        self.dtype = TORCH_DTYPE[wl.dtype]
        # capacity = rows after prefill + generated tokens + room for the steps
        self.cap = [sk.compressed_len(p, t, n, g, wl.w, layer, wl.l0) + extra_rows
                    for p, t, n, g in zip(wl.P, wl.T, wl.N, wl.G)]
        off = np.zeros(wl.B + 1, dtype=np.int64)
        off[1:] = np.cumsum(self.cap)
        self.cache_off = torch.from_numpy(off).to(device)
        rows = int(off[-1])
        shape = (rows * wl.H_kv * wl.d,)
        self.k = torch.zeros(shape, dtype=self.dtype, device=device)
        self.v = torch.zeros(shape, dtype=self.dtype, device=device)
        self.len = torch.zeros(wl.B, dtype=torch.int32, device=device)

    def block(self, t: torch.Tensor, b: int) -> torch.Tensor:
        """Request b's [H_kv, cap_b, d] view of a cache tensor."""
        off = self.cache_off.cpu().numpy()
        H, d = self.wl.H_kv, self.wl.d
        return t[off[b] * H * d: off[b + 1] * H * d].view(H, self.cap[b], d)

    def request_rows(self, b: int, n: int | None = None):
        """Request b's first n (default len[b]) cached rows, token-major
        [n, H_kv, d] float64 numpy, keys and values."""
        if n is None:
            n = int(self.len[b].item())
        k = self.block(self.k, b)[:, :n].permute(1, 0, 2)
        v = self.block(self.v, b)[:, :n].permute(1, 0, 2)
        return f64(k), f64(v)


def prefill_packed(wl: inputs.Workload, layer: int, device="cuda"):
    """Packed token-major prefill keys/values [sum S_b, H_kv, d], full_off."""
    ks, vs = zip(*[inputs.prefill_kv(wl, layer, b) for b in range(wl.B)])
    off = np.zeros(wl.B + 1, dtype=np.int64)
    off[1:] = np.cumsum(wl.full_rows())
    k = torch.cat(ks).to(device)
    v = torch.cat(vs).to(device)
    return k, v, torch.from_numpy(off).to(device), ks, vs


def lengths_dev(wl: inputs.Workload, device="cuda"):
    t = lambda x: torch.tensor(x, dtype=torch.int32, device=device)  # noqa: E731
    return t(wl.P), t(wl.T), t(wl.N)


def gpu_prefill(wl: inputs.Workload, layer: int, extra_rows: int, gate_scale: float = 1.0,
                device="cuda"):
    """GPU path: pool the prefill of every request into a fresh cache, then
    write the G[b] already-generated tokens (synthetic history) after it."""
    sk = lib()
    L = GpuLayer(wl, layer, extra_rows, device)
    k, v, full_off, ks, vs = prefill_packed(wl, layer, device)
    P, T, N = lengths_dev(wl, device)
    gate = torch.from_numpy(inputs.gate(wl, layer, gate_scale)).to(device)
    sk.pool(k, v, full_off, P, T, N, gate, L.k, L.v, L.cache_off, L.len, wl.w, layer, wl.l0)
    if max(wl.G) > 0:
        _place_generated(wl, layer, L)
    return L, (ks, vs, gate)


def _place_generated(wl, layer, L: GpuLayer):
    """Write generated-token rows straight into the cache blocks (synthetic
    history before the first checked step) and advance len."""
    lens = L.len.cpu().numpy()
    for b in range(wl.B):
        g = wl.G[b]
        if g == 0:
            continue
        kg, vg = inputs.generated_kv(wl, layer, b)
        L.block(L.k, b)[:, lens[b]:lens[b] + g] = kg.to(L.device).permute(1, 0, 2)
        L.block(L.v, b)[:, lens[b]:lens[b] + g] = vg.to(L.device).permute(1, 0, 2)
    L.len += torch.tensor(wl.G, dtype=torch.int32, device=L.device)


def oracle_prefill(oracle, wl: inputs.Workload, layer: int, extra_rows: int, ks, vs, gate):
    """Oracle path for the same inputs: per request [cap, H_kv, d] float64
    caches and row counts."""
    store = oracle.STORE_F32 if wl.dtype == "f32" else oracle.STORE_BF16
    caches = []
    for b in range(wl.B):
        Ko, Vo = oracle.pool_request(f64(ks[b]), f64(vs[b]), wl.P[b], wl.T[b], wl.N[b],
                                     f64(gate), wl.w, layer, wl.l0, storage=store)
        n = Ko.shape[0]
        cap = n + wl.G[b] + extra_rows
        Kc = np.zeros((cap, wl.H_kv, wl.d)); Vc = np.zeros_like(Kc)
        Kc[:n], Vc[:n] = Ko, Vo
        if wl.G[b]:
            kg, vg = inputs.generated_kv(wl, layer, b)
            kg, vg = f64(kg), f64(vg)
            for j in range(wl.G[b]):
                n = oracle.append_request(Kc, Vc, n, kg[j], vg[j])
        caches.append([Kc, Vc, n])
    return caches
