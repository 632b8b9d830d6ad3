"""The C ABI driven from a plain C program on the GPU (tests/c/compress_from_c.c): its retained slots
and compacted rows equal those of the Python binding on the same inputs, and its selection matches the
oracle."""
import os

import numpy as np
import pytest

from oracle import stepkv_oracle as O
import stepkv_testlib as TL
from test_cpu_abi import _build_c_program

pytestmark = pytest.mark.gpu

L, HKV, HQ, D, T, W, NSTEPS, NSAL = 2, 2, 8, 64, 1000, 16, 5, 2


def test_c_program_compress_matches_binding_and_oracle(tmp_path):
    import subprocess
    import torch
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    from paper_2609_22158_gb300 import binding as B
    exe = _build_c_program(tmp_path)
    out = subprocess.run([str(exe), "gpu", str(tmp_path)], check=True, capture_output=True, text=True).stdout
    n_kept = int(out.split()[1])
    rd = lambda name, dt: np.fromfile(os.path.join(tmp_path, name), dtype=dt)
    K = rd("K.bin", np.uint16).reshape(L, HKV, T, D)
    V = rd("V.bin", np.uint16).reshape(L, HKV, T, D)
    Q = rd("Q.bin", np.uint16).reshape(NSAL, HQ, W, D)
    step_id = rd("step_id.bin", np.int32)
    prot = rd("prot.bin", np.uint8)
    sig = rd("signals.bin", np.float32).reshape(4, NSTEPS)
    kept_c = rd("kept.bin", np.int32)
    kout_c = rd("K_out_layer1.bin", np.uint16).reshape(HKV, n_kept, D)
    assert kept_c.shape[0] == n_kept
    # the same inputs through the Python binding
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    Kd = [TL.bf16_dev(K[l]) for l in range(L)]
    Vd = [TL.bf16_dev(V[l]) for l in range(L)]
    Qd = [TL.bf16_dev(Q[i]) for i in range(NSAL)]
    reuse = np.zeros(NSTEPS, np.float32)
    steps = B.StepSignals(dev(sig[0]), dev(sig[1]), dev(sig[2]), dev(reuse), dev(sig[3]),
                          torch.empty(NSTEPS, dtype=torch.float32, device="cuda"))
    out_b = B.SelectOutputs.allocate(T, NSTEPS, T, "cuda", full=False)
    Ko = [torch.empty((HKV, T, D), dtype=torch.bfloat16, device="cuda") for _ in range(L)]
    Vo = [torch.empty((HKV, T, D), dtype=torch.bfloat16, device="cuda") for _ in range(L)]
    prob = B.Problem(Kd, Vd, Qd, T, dev(step_id), dev(prot), steps, B.budget_ratio(1, 4), Ko, Vo, out_b)
    st = B.stepkv_compress([prob], B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    assert int(out_b.n_kept.item()) == n_kept
    assert np.array_equal(out_b.kept_idx[:n_kept].cpu().numpy(), kept_c)
    assert np.array_equal(TL.bits_of(Ko[1][:, :n_kept]), kout_c)
    assert np.array_equal(kout_c, K[1][:, kept_c])
    # and the oracle on the same inputs
    ref = O.compress([K[l] for l in range(L - NSAL, L)], [Q[i] for i in range(NSAL)], step_id, prot, sig[0], sig[1],
                     sig[2], sig[3], reuse, TL.oracle_params(B.Params()), "ratio", num=1, den=4)
    TL.compare_kept(kept_c.astype(np.int64), ref)
