"""The usage example in README.md runs as written (on a GPU), and its
decode step matches the oracle."""
import os
import re

import pytest

from tests import harness as H

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_readme_example_runs(oracle):
    H.require_gpu()
    H.lib()  # builds the library if needed
    text = open(os.path.join(ROOT, "README.md")).read()
    blocks = re.findall(r"```python\n(.*?)```", text, re.S)
    assert blocks, "README.md has no python example"
    env = {}
    exec(compile(blocks[0], "README.md", "exec"), env)
    sk = env["sk"]
    assert sk.check_device_error() == sk.OK
    # the step's output against the oracle on the example's own cache
    import numpy as np
    lens = env["length"].cpu().numpy()
    cap, H_kv, d = env["cap"], env["H_kv"], env["d"]
    kc = env["k_cache"].view(-1, d)
    vc = env["v_cache"].view(-1, d)
    offs = [0]
    for c in cap:
        offs.append(offs[-1] + c)
    for b in range(env["B"]):
        n = int(lens[b])
        blk = lambda t: t[offs[b] * H_kv:(offs[b] + cap[b]) * H_kv].view(H_kv, cap[b], d)[:, :n]  # noqa: E731
        K = H.f64(blk(kc).permute(1, 0, 2))
        V = H.f64(blk(vc).permute(1, 0, 2))
        ref = oracle.decode_attn_request(H.f64(env["q"][b]), K, V, storage=oracle.STORE_BF16)
        H.assert_close(H.f64(env["out"][b]), np.asarray(ref), "bf16", f"request {b}")
