"""Failure detection on the GPU without a fault: the saliency kernel's cross-CTA wait is made to run out
(its second pass looks for a flag value no CTA publishes), the kernel reports STEPKV_ETIMEOUT through
the status word and returns, and the same context then computes correct results."""
import time

import numpy as np
import pytest

from oracle import stepkv_oracle as O
from paper_2609_22158_gb300 import workload as wl
import stepkv_testlib as TL

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    import torch
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    from paper_2609_22158_gb300 import binding, build
    build.build_library()
    binding.load_library()
    return binding


@pytest.mark.parametrize("d", [64, 128])
def test_saliency_wait_runs_out_and_context_stays_usable(B, d):
    import torch
    tr = wl.custom(61 + d, L=3, Hq=8, Hkv=2, d=d, T=2500, W=32, n_steps=7)
    Ks = [TL.bf16_dev(tr.keys(l)) for l in tr.sal_layer_ids()]
    Qs = [TL.bf16_dev(tr.queries(l)) for l in tr.sal_layer_ids()]
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    B.stepkv_selftest_score_timeout(Ks, Qs, tr.shape.T, 2_000_000, status)  # 2 ms limit
    torch.cuda.synchronize()
    elapsed = time.perf_counter() - t0
    assert status.item() == B.STEPKV_ETIMEOUT
    assert elapsed < 0.5, elapsed  # the wait gave up after its limit, well before the 1 s default
    # the same context, the same stream: a normal call computes the oracle's saliency
    st2 = torch.zeros(1, dtype=torch.int32, device="cuda")
    sal = B.stepkv_score(Ks, Qs, tr.shape.T, status=st2)
    torch.cuda.synchronize()
    assert st2.item() == 0
    for i, l in enumerate(tr.sal_layer_ids()):
        ref = O.window_attention_saliency(tr.keys(l), tr.queries(l))
        TL.assert_close(sal[i].cpu().numpy(), ref, f"saliency layer {l} after the timeout")


def test_selftest_rejects_bad_limits(B):
    import torch
    tr = wl.custom(5, L=1, Hq=8, Hkv=2, d=64, T=600, W=16, n_steps=3, n_sal_layers=1)
    Ks = [TL.bf16_dev(tr.keys(0))]
    Qs = [TL.bf16_dev(tr.queries(0))]
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for bad in (0, 999, 2_000_000_000):
        with pytest.raises(RuntimeError):
            B.stepkv_selftest_score_timeout(Ks, Qs, tr.shape.T, bad, status)
    torch.cuda.synchronize()
    assert status.item() == 0
