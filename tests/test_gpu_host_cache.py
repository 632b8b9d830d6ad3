"""Caches in page-locked host memory (kv_location / out_location = STEPKV_MEM_HOST): the compaction
reads and writes the retained rows across the CPU-GPU link, the saliency stage reads device copies of
the saliency layers' K.  Every output must equal the all-device pass on the same inputs bit for bit
(same saliency inputs, same kernels), and the oracle on the selection."""
import ctypes
import types

import numpy as np
import pytest

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


def _traj():
    return wl.custom(41, L=5, Hq=8, Hkv=2, d=128, T=3000, W=32, n_steps=9, budget=wl.Budget.ratio(1, 5))


def _device_run(B, g):
    import torch
    prob = g.problem()
    st = B.stepkv_compress([prob], B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    n = int(g.out.n_kept.item())
    return n, g.out.kept_idx[:n].clone(), [k[:, :n].clone() for k in g.K_out], [v[:, :n].clone() for v in g.V_out]


@pytest.mark.parametrize("kv_host,out_host", [(True, False), (True, True), (False, True)])
def test_host_resident_cache_matches_device_pass(B, kv_host, out_host):
    import torch
    tr = _traj()
    g = TL.GpuTraj(tr, kept_cap=tr.shape.T)
    n_ref, kept_ref, Kref, Vref = _device_run(B, g)
    s = tr.shape
    cap = g.kept_cap
    Kh = [k.cpu().pin_memory() for k in g.K] if kv_host else g.K
    Vh = [v.cpu().pin_memory() for v in g.V] if kv_host else g.V
    mk = (lambda: torch.zeros((s.Hkv, cap, s.d), dtype=torch.bfloat16).pin_memory()) if out_host else \
        (lambda: torch.zeros((s.Hkv, cap, s.d), dtype=torch.bfloat16, device="cuda"))
    K_out = [mk() for _ in range(s.L)]
    V_out = [mk() for _ in range(s.L)]
    out = B.SelectOutputs.allocate(s.T, tr.n_steps, cap, "cuda")
    sid_out = torch.full((cap,), -7, dtype=torch.int32, device="cuda")
    pos_out = torch.full((cap,), -7, dtype=torch.int32, device="cuda")
    K_sal = [g.K[l] for l in tr.sal_layer_ids()] if kv_host else None
    prob = B.Problem(Kh, Vh, g.Q, s.T, g.step_id, g.prot, g.steps(), g.budget(), K_out, V_out, out, pos_in=g.pos,
                     step_id_out=sid_out, pos_out=pos_out,
                     kv_location=B.STEPKV_MEM_HOST if kv_host else B.STEPKV_MEM_DEVICE,
                     out_location=B.STEPKV_MEM_HOST if out_host else B.STEPKV_MEM_DEVICE, K_sal=K_sal)
    st = B.stepkv_compress([prob], B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    n = int(out.n_kept.item())
    assert n == n_ref
    assert torch.equal(out.kept_idx[:n], kept_ref)
    for l in range(s.L):
        assert torch.equal(K_out[l][:, :n].cuda(), Kref[l])
        assert torch.equal(V_out[l][:, :n].cuda(), Vref[l])
    kept = kept_ref.long()
    assert torch.equal(sid_out[:n], g.step_id.index_select(0, kept))
    assert torch.equal(pos_out[:n], g.pos.index_select(0, kept))
    TL.check_select_outputs(types.SimpleNamespace(out=out, tr=tr, reuse_out=g.reuse_out),
                            TL.run_oracle(tr, TL.oracle_params(B.Params())))


def test_host_resident_cache_in_place(B):
    """Hole filling inside a host-resident cache: rows [0, n) of every layer end up holding the retained
    rows (as a set, each row's original slot given by pos_out), moved over the CPU-GPU link."""
    import torch
    tr = _traj()
    g = TL.GpuTraj(tr, kept_cap=tr.shape.T)
    n_ref, kept_ref, _, _ = _device_run(B, g)
    s = tr.shape
    Kh = [k.cpu().pin_memory() for k in g.K]
    Vh = [v.cpu().pin_memory() for v in g.V]
    K0 = [TL.bits_of(k) for k in g.K]
    V0 = [TL.bits_of(v) for v in g.V]
    out = B.SelectOutputs.allocate(s.T, tr.n_steps, s.T, "cuda")
    sid_out = torch.empty(s.T, dtype=torch.int32, device="cuda")
    pos_out = torch.empty(s.T, dtype=torch.int32, device="cuda")
    prob = B.Problem(Kh, Vh, g.Q, s.T, g.step_id, g.prot, g.steps(), g.budget(), Kh, Vh, out, pos_in=g.pos,
                     step_id_out=sid_out, pos_out=pos_out, kv_location=B.STEPKV_MEM_HOST,
                     out_location=B.STEPKV_MEM_HOST, K_sal=[g.K[l] for l in tr.sal_layer_ids()])
    st = B.stepkv_compress([prob], B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    n = int(out.n_kept.item())
    assert n == n_ref and torch.equal(out.kept_idx[:n], kept_ref)
    kept = kept_ref.cpu().numpy().astype(np.int64)
    slot_of_pos = {int(x): i for i, x in enumerate(tr.pos)}
    src = np.array([slot_of_pos[int(x)] for x in pos_out[:n].cpu().numpy()], np.int64)
    assert np.array_equal(np.sort(src), kept)
    below = kept[kept < n]
    assert np.array_equal(src[below], below)
    for l in range(s.L):
        assert np.array_equal(TL.bits_of(Kh[l][:, :n]), K0[l][:, src])
        assert np.array_equal(TL.bits_of(Vh[l][:, :n]), V0[l][:, src])


def test_host_location_rejects_other_memory(B):
    """A cache declared host-resident must be page-locked host memory: device or pageable pointers are
    refused on the host (STEPKV_EINVAL) before anything is enqueued."""
    import torch
    tr = _traj()
    g = TL.GpuTraj(tr, kept_cap=tr.shape.T)
    prob = g.problem()
    c = prob.c()
    lib = B.load_library()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    arr = (B.CProblem * 1)(c)
    need = int(lib.stepkv_compress_workspace_size(arr, 1))
    ws = torch.empty(need + 256, dtype=torch.uint8, device="cuda")
    wp = (ws.data_ptr() + 255) & ~255
    cp = B.Params().c()
    s = torch.cuda.current_stream().cuda_stream
    # device pointers declared host-resident
    sal = (ctypes.c_void_p * 3)(*[g.K[l].data_ptr() for l in tr.sal_layer_ids()])
    bad = B.CProblem.from_buffer_copy(c)
    bad.kv_location = B.STEPKV_MEM_HOST
    bad.K_sal = ctypes.cast(sal, ctypes.c_void_p)
    arr = (B.CProblem * 1)(bad)
    assert lib.stepkv_compress(arr, 1, ctypes.byref(cp), wp, need, st.data_ptr(), s) == B.STEPKV_EINVAL
    # host-resident without the device copies of the saliency layers
    bad.K_sal = None
    arr = (B.CProblem * 1)(bad)
    assert lib.stepkv_compress(arr, 1, ctypes.byref(cp), wp, need, st.data_ptr(), s) == B.STEPKV_EINVAL
    # pageable host memory declared as the output location
    pageable = [np.zeros(tr.shape.Hkv * tr.shape.T * tr.shape.d, np.uint16) for _ in range(2 * tr.shape.L)]
    outs = (ctypes.c_void_p * tr.shape.L)(*[a.ctypes.data for a in pageable[:tr.shape.L]])
    outs_v = (ctypes.c_void_p * tr.shape.L)(*[a.ctypes.data for a in pageable[tr.shape.L:]])
    bad = B.CProblem.from_buffer_copy(c)
    bad.out_location = B.STEPKV_MEM_HOST
    bad.K_out = ctypes.cast(outs, ctypes.c_void_p)
    bad.V_out = ctypes.cast(outs_v, ctypes.c_void_p)
    arr = (B.CProblem * 1)(bad)
    assert lib.stepkv_compress(arr, 1, ctypes.byref(cp), wp, need, st.data_ptr(), s) == B.STEPKV_EINVAL
    # an unknown location
    bad = B.CProblem.from_buffer_copy(c)
    bad.kv_location = 7
    arr = (B.CProblem * 1)(bad)
    assert lib.stepkv_compress(arr, 1, ctypes.byref(cp), wp, need, st.data_ptr(), s) == B.STEPKV_EINVAL
    torch.cuda.synchronize()
    assert st.item() == 0


def test_host_resident_batch_of_trajectories(B):
    """Several host-resident trajectories in one call (one shared saliency launch, one compaction
    launch): each equals its own all-device pass."""
    import torch
    trs = [wl.custom(71 + i, L=3, Hq=8, Hkv=2, d=64, T=T, W=16, n_steps=4 + i, budget=wl.Budget.ratio(1, 4))
           for i, T in enumerate((900, 1500, 2300))]
    refs, probs, outs = [], [], []
    for tr in trs:
        g = TL.GpuTraj(tr, kept_cap=tr.shape.T)
        refs.append(_device_run(B, g))
        s = tr.shape
        Kh = [k.cpu().pin_memory() for k in g.K]
        Vh = [v.cpu().pin_memory() for v in g.V]
        K_out = [torch.zeros((s.Hkv, s.T, s.d), dtype=torch.bfloat16).pin_memory() for _ in range(s.L)]
        V_out = [torch.zeros((s.Hkv, s.T, s.d), dtype=torch.bfloat16).pin_memory() for _ in range(s.L)]
        out = B.SelectOutputs.allocate(s.T, tr.n_steps, s.T, "cuda")
        probs.append(B.Problem(Kh, Vh, g.Q, s.T, g.step_id, g.prot, g.steps(), g.budget(), K_out, V_out, out,
                               pos_in=g.pos, kv_location=B.STEPKV_MEM_HOST, out_location=B.STEPKV_MEM_HOST,
                               K_sal=[g.K[l] for l in tr.sal_layer_ids()]))
        outs.append((out, K_out, V_out))
    st = B.stepkv_compress(probs, B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    for (n_ref, kept_ref, Kref, Vref), (out, K_out, V_out) in zip(refs, outs):
        n = int(out.n_kept.item())
        assert n == n_ref and torch.equal(out.kept_idx[:n], kept_ref)
        for l in range(len(K_out)):
            assert torch.equal(K_out[l][:, :n].cuda(), Kref[l])
            assert torch.equal(V_out[l][:, :n].cuda(), Vref[l])
