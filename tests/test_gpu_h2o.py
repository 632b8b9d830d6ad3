"""GPU parity of the accumulated-attention (H2O-style) token saliency against the CPU oracle, through the
C ABI: stepkv_decode_h2o adds every key's group-mean softmax weight to caller-owned mass rows at each decode
read (Sec. 4.2: T_i may come from an existing token-level importance estimator), and the accumulated rows
then drive the selection as its saliency rows.

Tolerance: masses element by element within 2e-3 relative (masses below 1e-30 compared absolutely: the
kernel's exponential flushes results below 2^-126); the decode outputs must equal stepkv_decode's bit for bit.
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


def _bits(rng, shape, scale=1.0):
    return wl.f32_to_bf16_bits(rng.standard_normal(shape).astype(np.float32) * np.float32(scale))


H2O_CASES = [
    # Hkv, G, d, n, rows, layers, reads, key scale
    (2, 4, 128, 1000, 1100, 2, 3, 1.0),   # ragged last split, capacity above n
    (8, 4, 128, 8272, 8272, 1, 2, 1.0),   # the incremental loop's compacted cache shape
    (2, 5, 128, 700, 700, 1, 2, 1.0),     # G = 5
    (1, 8, 64, 513, 600, 1, 3, 3.0),      # G = 8, d = 64, peaky softmax
    (4, 1, 64, 2049, 2100, 1, 1, 1.0),    # no grouping
    (2, 2, 64, 1, 1, 1, 2, 1.0),          # a single key takes all the mass
]


@pytest.mark.parametrize("Hkv,G,d,n,rows,L,reads,ks", H2O_CASES)
def test_h2o_mass_matches_oracle(B, Hkv, G, d, n, rows, L, reads, ks):
    import torch
    rng = np.random.default_rng(300 + n + d + G)
    Ks = [_bits(rng, (Hkv, rows, d), ks) for _ in range(L)]
    Vs = [_bits(rng, (Hkv, rows, d)) for _ in range(L)]
    Kd, Vd = [TL.bf16_dev(x) for x in Ks], [TL.bf16_dev(x) for x in Vs]
    mass = [torch.zeros((Hkv, rows + 5), dtype=torch.float32, device="cuda") for _ in range(L)]
    ref = [np.zeros((Hkv, n)) for _ in range(L)]
    st = B.new_status()
    for r in range(reads):
        qs = [_bits(rng, (Hkv * G, d)) for _ in range(L)]
        qd = [TL.bf16_dev(x) for x in qs]
        out = B.stepkv_decode_h2o(qd, Kd, Vd, n, mass, status=st)
        plain = B.stepkv_decode(qd, Kd, Vd, n, status=st)
        torch.cuda.synchronize()
        assert st.item() == 0
        for l in range(L):
            assert torch.equal(out[l], plain[l]), "decode output differs from stepkv_decode"
            ref[l] += O.decode_attention_mass(qs[l], Ks[l][:, :n])
    for l in range(L):
        g = mass[l].cpu().numpy()
        TL.assert_close(g[:, :n], ref[l], f"accumulated mass layer {l}", floor=1e-30)
        assert np.all(g[:, n:] == 0.0), "mass written past n"
        assert np.allclose(g[:, :n].sum(axis=1), reads, rtol=1e-5)


def test_h2o_n_on_device_and_determinism(B):
    import torch
    rng = np.random.default_rng(8)
    Hkv, G, d, rows, n = 2, 4, 128, 1500, 1234
    q = [TL.bf16_dev(_bits(rng, (Hkv * G, d)))]
    K = [TL.bf16_dev(_bits(rng, (Hkv, rows, d)))]
    V = [TL.bf16_dev(_bits(rng, (Hkv, rows, d)))]
    m1 = [torch.zeros((Hkv, rows), dtype=torch.float32, device="cuda")]
    m2 = [torch.zeros((Hkv, rows), dtype=torch.float32, device="cuda")]
    B.stepkv_decode_h2o(q, K, V, n, m1)
    B.stepkv_decode_h2o(q, K, V, torch.tensor([n], dtype=torch.int32, device="cuda"), m2)
    torch.cuda.synchronize()
    assert torch.equal(m1[0], m2[0])


def test_h2o_mass_drives_selection(B):
    """Masses accumulated over 4 decode reads of a 3-layer cache become the selection's saliency rows
    (T_i = their mean over layers and KV heads), at the Table H weights and with the saliency term alone
    (alpha = 1, beta = 0); every selection output is compared with the oracle's boundary on the oracle's
    masses."""
    import torch
    tr = wl.custom(71, L=3, Hq=16, Hkv=4, d=128, T=3000, W=32, n_steps=7, budget=wl.Budget.ratio(1, 5))
    s = tr.shape
    Ks = [tr.keys(l) for l in range(s.L)]
    Vs = [tr.values(l) for l in range(s.L)]
    Kd, Vd = [TL.bf16_dev(x) for x in Ks], [TL.bf16_dev(x) for x in Vs]
    mass = torch.zeros((s.L, s.Hkv, s.T), dtype=torch.float32, device="cuda")
    ref = [np.zeros((s.Hkv, s.T)) for _ in range(s.L)]
    qs_all = wl.decode_queries(72, s.L, s.Hq, s.d, 4)
    for r in range(4):
        qs = [qs_all[r, l] for l in range(s.L)]
        B.stepkv_decode_h2o([TL.bf16_dev(x) for x in qs], Kd, Vd, s.T, [mass[l] for l in range(s.L)])
        for l in range(s.L):
            ref[l] += O.decode_attention_mass(qs[l], Ks[l])
    torch.cuda.synchronize()
    for alpha, beta in ((0.2, 0.8), (1.0, 0.0)):
        p = B.Params()
        p.alpha, p.beta = alpha, beta
        g = TL.GpuTraj(tr)
        g.out = B.SelectOutputs.allocate(s.T, tr.n_steps, s.T, "cuda")
        st = B.new_status()
        B.stepkv_select(mass.view(s.L * s.Hkv, s.T), g.step_id, g.prot, g.steps(), p, g.budget(), g.out, status=st)
        torch.cuda.synchronize()
        assert st.item() == 0
        b = tr.budget
        out = O.stepkv_boundary(ref, tr.step_id, tr.prot, tr.valid, tr.gain, tr.red, tr.obs_sim, tr.reuse,
                                TL.oracle_params(p), b.mode, b.num, b.den, b.count)
        assert TL.check_select_outputs(g, out) == 0
