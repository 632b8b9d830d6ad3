"""stepkv_compress inside a CUDA graph: captured once, then replayed with new data in the same buffers.

The saliency kernel's cross-CTA waits compare flags against a per-launch token.  A replayed launch has the
same kernel parameters as the captured one, so the token also mixes in a per-workspace epoch that the
kernel advances itself; without it a replay would find the previous replay's flags already set and start
its second pass on stale partials.  Each replay here runs on different keys, queries and step signals and
must match the oracle like a direct call.
"""
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


def _load(g, tr):
    """Copy trajectory tr (same shapes as g's) into g's device buffers."""
    import torch
    for l in range(tr.shape.L):
        g.K[l].copy_(TL.bf16_dev(tr.keys(l)))
        g.V[l].copy_(TL.bf16_dev(tr.values(l)))
    for i, l in enumerate(tr.sal_layer_ids()):
        g.Q[i].copy_(TL.bf16_dev(tr.queries(l)))
    for name, arr in (("step_id", tr.step_id), ("prot", tr.prot), ("pos", tr.pos), ("valid", tr.valid),
                      ("gain", tr.gain), ("red", tr.red), ("obs_sim", tr.obs_sim), ("reuse_in", tr.reuse)):
        getattr(g, name).copy_(torch.from_numpy(arr).cuda())
    g.tr = tr


def test_compress_graph_replay(B):
    import torch
    trs = [wl.custom(600 + i, L=4, Hq=32, Hkv=8, d=128, T=6000, W=64, n_steps=8,
                     budget=wl.Budget.ratio(1, 10)) for i in range(3)]
    g = TL.GpuTraj(trs[0])
    prob = g.problem()
    p = B.Params()
    ws = torch.empty(B.stepkv_workspace_size([prob]) + 512, dtype=torch.uint8, device="cuda")
    status = B.new_status()
    stream = torch.cuda.Stream()
    # one direct call first (loads the library, sets the kernels' shared-memory limits)
    with torch.cuda.stream(stream):
        B.stepkv_compress([prob], p, ws=ws, status=status, stream=stream)
    torch.cuda.synchronize()
    assert status.item() == 0
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream, capture_error_mode="thread_local"):
        B.stepkv_compress([prob], p, ws=ws, status=status, stream=stream)
    torch.cuda.synchronize()
    op = TL.oracle_params(p)
    kept_sets = []
    for rep in range(2):
        for tr in trs:
            _load(g, tr)
            torch.cuda.synchronize()
            with torch.cuda.stream(stream):
                graph.replay()
            torch.cuda.synchronize()
            assert status.item() == 0, status.item()
            out = TL.run_oracle(tr, op)
            TL.check_select_outputs(g, out)
            n = int(g.out.n_kept.item())
            gk = g.out.kept_idx[:n].cpu().numpy()
            for l in (0, tr.shape.L - 1):
                assert np.array_equal(TL.bits_of(g.K_out[l])[:, :n], O.compact_rows(tr.keys(l), gk))
                assert np.array_equal(TL.bits_of(g.V_out[l])[:, :n], O.compact_rows(tr.values(l), gk))
            kept_sets.append(gk.copy())
    # replays of the same data give the same retained set (bit-exact, deterministic)
    for i in range(3):
        assert np.array_equal(kept_sets[i], kept_sets[i + 3])
    assert not np.array_equal(kept_sets[0], kept_sets[1])
