"""Full-size parity on the batched ragged workload (16 trajectories, T ~ U(8K, 32K), 32 layers, key
outlier channels, budgets 5/10/20%) and the Qwen2.5-32B-shaped long horizon (64 layers, GQA 5,
W = 128, T = 65536, fixed budget 4096), in the launch configuration of the fused pass
(stepkv_compress over all trajectories in one call).

The saliency layers come from the seeded generator, so the oracle sees exactly the device inputs;
the other layers (compaction only) are device random tensors, checked bit-exact against an
index_select of the retained rows.  The oracle's saliency is computed once per trajectory and reused
across budgets.
"""
import os

import numpy as np
import pytest

from oracle import stepkv_oracle as O
from paper_2609_22158_gb300 import workload as wl
import stepkv_testlib as TL

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module")
def B():
    import torch
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    from paper_2609_22158_gb300 import binding, build
    build.build_library()
    binding.load_library()
    return binding


def _device_traj(tr, seed, kept_cap):
    import torch
    s = tr.shape
    gen = torch.Generator(device="cuda").manual_seed(seed)
    sal_ids = set(tr.sal_layer_ids())
    g = TL.GpuTraj.__new__(TL.GpuTraj)
    g.tr = tr
    g.L = s.L
    g.K = [TL.bf16_dev(tr.keys(l)) if l in sal_ids else
           torch.randn((s.Hkv, s.T, s.d), generator=gen, device="cuda", dtype=torch.bfloat16) for l in range(s.L)]
    g.V = [torch.randn((s.Hkv, s.T, s.d), generator=gen, device="cuda", dtype=torch.bfloat16) for _ in range(s.L)]
    g.Q = [TL.bf16_dev(tr.queries(l)) for l in tr.sal_layer_ids()]
    for nm, arr in (("step_id", tr.step_id), ("prot", tr.prot), ("pos", tr.pos), ("valid", tr.valid),
                    ("gain", tr.gain), ("red", tr.red), ("obs_sim", tr.obs_sim), ("reuse_in", tr.reuse)):
        setattr(g, nm, torch.from_numpy(arr).cuda())
    g.reuse_out = torch.empty_like(g.reuse_in)
    g.kept_cap = kept_cap
    return g


def _oracle_saliency(tr):
    return [O.window_attention_saliency(tr.keys(l), tr.queries(l)) for l in tr.sal_layer_ids()]


def _ragged_saliency_job(i):
    # runs in a spawned worker (no CUDA state): regenerate trajectory i and compute its saliency
    return _oracle_saliency(wl.ragged_batch()[i])


def _qwen_saliency_job(layer):
    tr = wl.qwen32b_64k()
    return O.window_attention_saliency(tr.keys(layer), tr.queries(layer))


def _spawn_map(fn, items):
    """The oracle in spawned worker processes (one BLAS thread each); spawn is safe after CUDA init."""
    import concurrent.futures as cf
    import multiprocessing as mp
    saved = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")}
    for k in saved:
        os.environ[k] = "1"
    try:
        workers = max(1, min(len(items), os.cpu_count() or 1))
        with cf.ProcessPoolExecutor(max_workers=workers, mp_context=mp.get_context("spawn")) as ex:
            return list(ex.map(fn, items))
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v


def _ragged_saliency_all(n):
    return _spawn_map(_ragged_saliency_job, list(range(n)))


def _oracle_boundary(tr, A, budget):
    p = TL.oracle_params(__import__("paper_2609_22158_gb300.binding", fromlist=["Params"]).Params())
    return O.stepkv_boundary(A, tr.step_id, tr.prot, tr.valid, tr.gain, tr.red, tr.obs_sim, tr.reuse, p,
                             budget.mode, budget.num, budget.den, budget.count)


def _check(g, out, layers=None):
    import torch
    swaps = TL.check_select_outputs(g, out)
    n = int(g.out.n_kept.item())
    kept = g.out.kept_idx[:n].long()
    for l in (range(g.tr.shape.L) if layers is None else layers):
        assert torch.equal(g.K_out[l][:, :n], g.K[l].index_select(1, kept))
        assert torch.equal(g.V_out[l][:, :n], g.V[l].index_select(1, kept))
    assert torch.equal(g.step_id_out[:n], g.step_id.index_select(0, kept))
    assert torch.equal(g.pos_out[:n], g.pos.index_select(0, kept))
    return swaps


def _bbudget(B, b):
    return B.budget_ratio(b.num, b.den) if b.mode == "ratio" else B.budget_count(b.count)


def test_batched_ragged_16_trajectories_full(B):
    import torch
    trs = wl.ragged_batch()
    assert len(trs) == 16
    gs = [_device_traj(tr, 3000 + i, tr.shape.T // 5 + 128) for i, tr in enumerate(trs)]
    A = _ragged_saliency_all(len(trs))
    total_swaps = 0
    for num, den in ((1, 10), (1, 20), (1, 5)):
        budget = wl.Budget.ratio(num, den)
        probs = [g.problem(_bbudget(B, budget)) for g in gs]
        st = B.stepkv_compress(probs, B.Params())
        torch.cuda.synchronize()
        assert st.item() == 0, (num, den)
        for g, tr, a in zip(gs, trs, A):
            out = _oracle_boundary(tr, a, budget)
            # compaction of every layer once (10%), the selection outputs for every budget
            total_swaps += _check(g, out, layers=None if (num, den) == (1, 10) else tr.sal_layer_ids())
    print(f"batched ragged swaps: {total_swaps}")


def test_qwen32b_64k_long_horizon_full(B):
    import torch
    tr = wl.qwen32b_64k()
    s = tr.shape
    assert (s.L, s.Hq, s.Hkv, s.T, s.W) == (64, 40, 8, 65536, 128)
    g = _device_traj(tr, 4000, 4096 + 16 + 128)
    prob = g.problem()
    st = B.stepkv_compress([prob], B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    out = _oracle_boundary(tr, _spawn_map(_qwen_saliency_job, list(tr.sal_layer_ids())), tr.budget)
    assert out["B"] == 4096
    swaps = _check(g, out)
    assert int(g.out.n_kept.item()) == 16 + 128 + 4096
    print(f"qwen 64K swaps: {swaps}")
