"""GPU parity of decode attention over a (compacted) cache against the CPU oracle, through the C ABI.

Tolerance: element by element, |gpu - oracle| <= 2e-3 x max(|oracle|, 1e-3 x m), where m is the magnitude
of the weighted sum's terms, sum_j p_j |V[j]| (stepkv_testlib.DECODE_FLOOR).  The GPU computes logits in
fp32 from exact bf16 products, exponentials with the MUFU ex2 and fp32 sums over at most a few thousand
weighted rows, so its error is orders of magnitude below that.
"""
import numpy as np
import pytest

from oracle import stepkv_oracle as O
from paper_2609_22158_gb300 import workload as wl
import stepkv_testlib as TL

pytestmark = pytest.mark.gpu
TOL = 2e-3


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


DECODE_CASES = [
    # Hkv, G, d, n, rows, layers, key scale
    (2, 4, 128, 1, 1, 1, 1.0),        # a single key: the output is that key's value row
    (2, 4, 128, 1000, 1000, 2, 1.0),  # ragged last split (1000 = 512 + 488)
    (8, 4, 128, 8272, 8272, 1, 1.0),  # the incremental loop's compacted cache (8192 budget + prefix/window)
    (2, 2, 64, 513, 600, 3, 2.0),     # d = 64, capacity stride above n, one key past a split
    (1, 8, 128, 777, 900, 1, 3.0),    # G = 8, peaky softmax
    (2, 5, 128, 300, 300, 1, 1.0),    # G = 5
    (4, 1, 64, 2049, 2100, 1, 1.0),   # no grouping
]


@pytest.mark.parametrize("Hkv,G,d,n,rows,L,ks", DECODE_CASES)
def test_decode_matches_oracle(B, Hkv, G, d, n, rows, L, ks):
    import torch
    rng = np.random.default_rng(100 + n + d + G)
    qs = [_bits(rng, (Hkv * G, d)) for _ in range(L)]
    Ks = [_bits(rng, (Hkv, rows, d), ks) for _ in range(L)]
    Vs = [_bits(rng, (Hkv, rows, d)) for _ in range(L)]
    st = B.new_status()
    out = B.stepkv_decode([TL.bf16_dev(x) for x in qs], [TL.bf16_dev(x) for x in Ks], [TL.bf16_dev(x) for x in Vs],
                          n, status=st)
    torch.cuda.synchronize()
    assert st.item() == 0
    for l in range(L):
        TL.assert_decode_close(out[l].cpu().numpy(), qs[l], Ks[l][:, :n], Vs[l][:, :n], f"layer {l}")


def test_decode_n_on_device_equals_host_n(B):
    import torch
    rng = np.random.default_rng(5)
    Hkv, G, d, rows, n = 2, 4, 128, 1200, 1100
    q = [TL.bf16_dev(_bits(rng, (Hkv * G, d)))]
    K = [TL.bf16_dev(_bits(rng, (Hkv, rows, d)))]
    V = [TL.bf16_dev(_bits(rng, (Hkv, rows, d)))]
    a = B.stepkv_decode(q, K, V, n)[0]
    b = B.stepkv_decode(q, K, V, torch.tensor([n], dtype=torch.int32, device="cuda"))[0]
    c = B.stepkv_decode(q, K, V, n)[0]
    torch.cuda.synchronize()
    assert torch.equal(a, b) and torch.equal(a, c)  # device-side n, and run-to-run determinism


def test_decode_n_above_capacity_sets_enospace(B):
    import torch
    rng = np.random.default_rng(6)
    Hkv, G, d, rows = 1, 4, 64, 300
    q = [TL.bf16_dev(_bits(rng, (Hkv * G, d)))]
    K = [TL.bf16_dev(_bits(rng, (Hkv, rows, d)))]
    V = [TL.bf16_dev(_bits(rng, (Hkv, rows, d)))]
    st = B.new_status()
    over = B.stepkv_decode(q, K, V, torch.tensor([rows + 7], dtype=torch.int32, device="cuda"), status=st)[0]
    full = B.stepkv_decode(q, K, V, rows)[0]
    torch.cuda.synchronize()
    assert st.item() == B.STEPKV_ENOSPACE
    assert torch.equal(over, full)  # clamped to the capacity


def test_decode_over_compacted_cache(B):
    """Compress a trajectory, then decode over K_out/V_out with n = n_kept read on the device."""
    import torch
    tr = wl.custom(51, L=2, Hq=8, Hkv=2, d=128, T=3000, W=32, n_steps=6, budget=wl.Budget.ratio(1, 5))
    g = TL.GpuTraj(tr)
    prob = g.problem()
    st = B.stepkv_compress([prob], B.Params())
    rng = np.random.default_rng(52)
    qs = [_bits(rng, (8, 128)) for _ in range(tr.shape.L)]
    out = B.stepkv_decode([TL.bf16_dev(x) for x in qs], g.K_out, g.V_out, g.out.n_kept, status=st)
    torch.cuda.synchronize()
    assert st.item() == 0
    n = int(g.out.n_kept.item())
    kept = g.out.kept_idx[:n].cpu().numpy()
    for l in range(tr.shape.L):
        TL.assert_decode_close(out[l].cpu().numpy(), qs[l], O.compact_rows(tr.keys(l), kept),
                               O.compact_rows(tr.values(l), kept), f"layer {l}")
