"""The build with device-side index checks (libkvlink_debug.so, KVLINK_DEBUG_CHECKS).

Its kernels check every work item, merge group, re-encode unit and fresh-row
destination against the plan's bounds before using it, and record a code in the device
status word instead of touching memory through a bad entry.  On valid plans the checks
must never fire and the results must be the release build's, bit for bit: every path
(per-layer linked prefill, the overlapped all-layers call, split KV ranges and their
merge, the paged pool, both cache layouts, zero-copy values) runs once in a child process bound to the
debug library and once here with the release library.
"""
import os
import subprocess
import sys

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
DEBUG_LIB = os.path.join(ROOT, "paper_2502_16002_gb300", "libkvlink_debug.so")

CASES = [(1, 0), (2, 0), (3, 0), (3, 1), (5, 0)]     # (workload, layout): workload 2 splits KV ranges

_CHILD = r"""
import sys, numpy as np, torch
sys.path.insert(0, {root!r}); sys.path.insert(0, {tests!r})
import workloads as W
from paper_2502_16002_gb300 import kvlink as K
from paper_2502_16002_gb300 import runtime as RT
dev = torch.device("cuda:0")
res = {{}}
for cfg_index, layout in {cases!r}:
    batch = W.draw_batch(W.get_config(cfg_index))
    n_layers = 2
    lp = RT.LinkedPrefill.from_batch(batch, device=dev, layout=layout)
    pk, pv, q, kn, vn = [], [], [], [], []
    for l in range(n_layers):
        a, b = W.pool_kv(batch, l); x, y, z = W.fresh_qkv(batch, l)
        for lst, arr in zip((pk, pv, q, kn, vn), (a, b, x, y, z)):
            lst.append(RT.bf16_from_bits(arr, dev))
    caches = [lp.empty_cache() for _ in range(n_layers)]
    outs = [torch.empty_like(x) for x in q]
    lp.linked_prefill_layers_overlapped(pk, pv, q, kn, vn, [c[0] for c in caches], [c[1] for c in caches], outs)
    ck, cv = lp.empty_cache(); o1 = torch.empty_like(q[0])
    lp.linked_prefill(pk[0], pv[0], q[0], kn[0], vn[0], ck, cv, o1)
    ck2 = lp.empty_cache()[0]; o2 = torch.empty_like(q[0])
    lp.linked_prefill(pk[0], pv[0], q[0], kn[0], vn[0], ck2, None, o2)     # zero-copy values
    torch.cuda.synchronize()
    assert K.kvlink_device_status() == 0, (cfg_index, layout, K.kvlink_device_status())
    for l in range(n_layers):
        res[f"{{cfg_index}}_{{layout}}_{{l}}_k"] = RT.bits_from_bf16(caches[l][0])
        res[f"{{cfg_index}}_{{layout}}_{{l}}_v"] = RT.bits_from_bf16(caches[l][1])
        res[f"{{cfg_index}}_{{layout}}_{{l}}_o"] = RT.bits_from_bf16(outs[l])
    res[f"{{cfg_index}}_{{layout}}_single_o"] = RT.bits_from_bf16(o1)
    res[f"{{cfg_index}}_{{layout}}_zero_copy_o"] = RT.bits_from_bf16(o2)
np.savez({out!r}, **res)
print("ok")
"""


def _run(lib, out, tmp):
    env = dict(os.environ)
    if lib:
        env["KVLINK_LIBRARY"] = lib
    else:
        env.pop("KVLINK_LIBRARY", None)
    script = _CHILD.format(root=ROOT, tests=os.path.dirname(os.path.abspath(__file__)), cases=CASES, out=out)
    r = subprocess.run([sys.executable, "-c", script], env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    return np.load(out)


def test_debug_build_gives_the_release_results(tmp_path):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    if not os.path.exists(DEBUG_LIB):
        pytest.skip("the debug library has not been built")
    dbg = _run(DEBUG_LIB, str(tmp_path / "debug.npz"), tmp_path)
    rel = _run(None, str(tmp_path / "release.npz"), tmp_path)
    assert sorted(dbg.files) == sorted(rel.files)
    for k in rel.files:
        assert np.array_equal(dbg[k], rel[k]), k
