"""GPU parity of the Sec. 4.1 field signals computed from evidence cues (stepkv_step_signals) against the
CPU oracle, through the C ABI, and the signals feeding the fused pass.

Tolerance: the signals are ratios of cue counts computed in fp32 (one division each), so they must agree
with the oracle's fp64 values within 1e-6 relative; a count outside [0, 64] or an unsorted cue list must set
STEPKV_EDATA and leave the affected values unwritten.
"""
import numpy as np
import pytest

from oracle import stepkv_oracle as O
from paper_2609_22158_gb300 import cues as C, workload as wl
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


def _dev(steps):
    import torch
    cues, cnt = C.pack_cues(steps)
    return torch.from_numpy(cues.view(np.int32)).cuda(), torch.from_numpy(cnt).cuda()


@pytest.mark.parametrize("n_steps,k0,seed", [(1, 0, 1), (2, 0, 2), (40, 0, 3), (40, 39, 4), (200, 150, 5)])
def test_step_signals_match_oracle(B, n_steps, k0, seed):
    import torch
    steps = wl.synthetic_cues(seed, n_steps)
    cues, cnt = _dev(steps)
    st = B.new_status()
    gain, red, obs_sim = B.stepkv_step_signals(cues, cnt, k0=k0, status=st)
    torch.cuda.synchronize()
    assert st.item() == 0
    og, orr, oo = O.step_signals([s[0] for s in steps], [s[1] for s in steps], [s[2] for s in steps], k0=k0)
    g, r, o = gain.cpu().numpy(), red.cpu().numpy(), obs_sim.cpu().numpy()
    assert np.all(np.isnan(g[:k0])) and np.all(np.isnan(r[:k0]))
    TL.assert_close(g[k0:], og[k0:], "gain", rtol=1e-6)
    TL.assert_close(r[k0:], orr[k0:], "red", rtol=1e-6)
    TL.assert_close(o, oo, "obs_sim", rtol=1e-6)


def test_step_signals_golden_table(B):
    """The hand-computed table of tests/golden/step_signals.txt (empty fields included)."""
    import os
    import torch
    parse = lambda x: [] if x == "-" else [int(v) for v in x.split(",")]
    steps, sig = [], []
    for line in open(os.path.join(os.path.dirname(__file__), "golden", "step_signals.txt")):
        if line.startswith("step "):
            _, _, th, act, obs = line.split()
            steps.append((parse(th), parse(act), parse(obs)))
        elif line.startswith("sig "):
            sig.append([float(v) for v in line.split()[2:]])
    sig = np.array(sig)
    cues, cnt = _dev(steps)
    gain, red, obs_sim = B.stepkv_step_signals(cues, cnt, k0=0)
    torch.cuda.synchronize()
    TL.assert_close(gain.cpu().numpy(), sig[:, 0], "gain", rtol=1e-6)
    TL.assert_close(red.cpu().numpy(), sig[:, 1], "red", rtol=1e-6)
    TL.assert_close(obs_sim.cpu().numpy(), sig[:, 2], "obs_sim", rtol=1e-6)


def test_step_signals_reject_unsorted_cues(B):
    import torch
    steps = wl.synthetic_cues(6, 10)
    cues, cnt = C.pack_cues(steps)
    cues[4, 0, [0, 1]] = cues[4, 0, [1, 0]]  # step 4's Thought no longer increasing
    st = B.new_status()
    gain, red, obs_sim = B.stepkv_step_signals(torch.from_numpy(cues.view(np.int32)).cuda(),
                                               torch.from_numpy(cnt).cuda(), k0=0, status=st)
    torch.cuda.synchronize()
    assert st.item() == B.STEPKV_EDATA
    g = gain.cpu().numpy()
    assert np.isnan(g[4:]).all() and np.isfinite(g[:4]).all()  # every target that compares with step 4


def test_signals_drive_the_fused_pass(B):
    """Cue-derived signals (gain, red, obs_sim from the kernel; valid from the workload) go straight into
    stepkv_compress; the oracle takes its own cue-derived signals."""
    import torch
    tr = wl.custom(91, L=3, Hq=8, Hkv=2, d=128, T=4000, W=32, n_steps=9, budget=wl.Budget.ratio(1, 6))
    steps = wl.synthetic_cues(92, tr.n_steps)
    cues, cnt = _dev(steps)
    g = TL.GpuTraj(tr)
    B.stepkv_step_signals(cues, cnt, k0=0, gain=g.gain, red=g.red, obs_sim=g.obs_sim)
    prob = g.problem()
    st = B.stepkv_compress([prob], B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    og, orr, oo = O.step_signals([s[0] for s in steps], [s[1] for s in steps], [s[2] for s in steps], k0=0)
    b = tr.budget
    Ks = [tr.keys(l) for l in tr.sal_layer_ids()]
    Qs = [tr.queries(l) for l in tr.sal_layer_ids()]
    out = O.compress(Ks, Qs, tr.step_id, tr.prot, tr.valid, og, orr, oo, tr.reuse, O.Params(), b.mode, b.num, b.den,
                     b.count)
    TL.check_select_outputs(g, out)
