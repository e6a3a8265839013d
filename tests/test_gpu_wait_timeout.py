"""The failure path of the bounded waits, driven on the GPU without a fault.

Every mbarrier wait in the attention kernels is bounded in time; when a bound runs out
the kernel records KVLINK_STATUS_WAIT_TIMEOUT in the device status word, drains its own
asynchronous work, frees its tensor memory and returns.  kvlink_selftest_wait_timeout
runs that same wait on a barrier nothing arrives at, with a short bound, so the expiry
path runs for real: no trap, no hang, and the context stays usable.  The test then checks
that later attention launches skip their work while the status is set (they return at
once instead of waiting out their own bounds) and that clearing the status restores
correct results.
"""
import time

import numpy as np
import pytest

import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from _gpu_common import check_query, run_layer  # noqa: E402


@pytest.fixture(scope="module")
def env():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_16002_gb300 import kvlink as K
    from paper_2502_16002_gb300 import runtime as RT

    return K, RT


def test_selftest_limit_is_validated(env):
    K, _ = env
    for bad in (0, 2001):
        with pytest.raises(K.KvlinkError) as e:
            K.kvlink_selftest_wait_timeout(bad, 0)
        assert e.value.code == K.KVLINK_EINVAL


def test_expired_wait_is_reported_and_later_launches_skip(env):
    K, RT = env
    dev = torch.device("cuda:0")
    batch = W.draw_batch(W.get_config(3))
    lp = RT.LinkedPrefill.from_batch(batch, device=dev)
    pk, pv = W.pool_kv(batch, 0)
    q, kn, vn = W.fresh_qkv(batch, 0)
    t = [RT.bf16_from_bits(a, dev) for a in (pk, pv, q, kn, vn)]
    ck, cv = lp.empty_cache()
    out = torch.empty(lp.fresh_shape(batch.cfg.h_q), dtype=torch.bfloat16, device=dev)
    lp.linked_prefill(*t, ck, cv, out)          # warm: every launch configured once
    torch.cuda.synchronize(dev)
    K.kvlink_clear_device_status()
    assert K.kvlink_device_status() == 0
    try:
        t0 = time.perf_counter()
        K.kvlink_selftest_wait_timeout(50, 0)
        torch.cuda.synchronize(dev)
        waited = time.perf_counter() - t0
        assert K.kvlink_device_status() == K.KVLINK_STATUS_WAIT_TIMEOUT
        assert 0.045 <= waited < 1.5, waited
        assert int(torch.arange(100, device=dev).sum().item()) == 4950    # the context still works
        # with the status set, the attention's CTAs return at once: a full workload-3 layer
        # finishes in well under one wait bound (2 s), and the status keeps its first code
        out.fill_(0)
        t0 = time.perf_counter()
        for _ in range(4):
            lp.suffix_attention(t[2], None, None, ck, cv, out)
        torch.cuda.synchronize(dev)
        assert time.perf_counter() - t0 < 0.5
        assert K.kvlink_device_status() == K.KVLINK_STATUS_WAIT_TIMEOUT
        # split ranges are merged inside the attention kernel, which did nothing: the output
        # was never written
        assert int(torch.count_nonzero(out.view(torch.int16)).item()) == 0
    finally:
        K.kvlink_clear_device_status()
    assert K.kvlink_device_status() == 0
    # re-armed: the same layer is correct again
    lp2, gk, gv, gout, inp = run_layer(RT, batch, 0, "fused")
    check_query(batch, 1, lp2, gk, gv, gout, inp)
    assert np.all(np.isfinite(gout))
