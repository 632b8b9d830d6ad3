"""stepkv_select_static_scratch against stepkv_select.

The static-scratch entry point serves callers that cannot allocate device memory at call time (device
memory reserved up front by a cache pool, no room for the synchronisation a free implies, no caching
allocator): it takes no workspace and uses a fixed scratch array in the library's device image.  It must
give the same selection as stepkv_select with a caller workspace, call after call.

The file name sorts last so that pytest collects it after every other GPU test: it has to pass both
alone and after the rest of the suite has used the device (and the library's other scratch).
"""
import ctypes

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


def _assert_close(a, b, what):
    """Within the parity tolerance on finite entries; -inf (protected priorities) at the same slots."""
    fin = np.isfinite(b)
    assert np.array_equal(np.isfinite(a), fin), f"{what}: non-finite entries differ"
    assert np.array_equal(a[~fin], b[~fin]), what
    if fin.any():
        TL.assert_close(a[fin], b[fin], what)


class _Case:
    """One trajectory's selection inputs on the device, plus two output sets (static, workspace)."""

    def __init__(self, B, tr, seed):
        import torch
        self.tr = tr
        rng = np.random.default_rng(seed)
        self.sal = torch.from_numpy((rng.random((3, tr.T)) * 2).astype(np.float32)).cuda()
        self.step_id = torch.from_numpy(tr.step_id).cuda()
        self.prot = torch.from_numpy(tr.prot).cuda()
        self.valid = torch.from_numpy(tr.valid).cuda()
        self.gain = torch.from_numpy(tr.gain).cuda()
        self.red = torch.from_numpy(tr.red).cuda()
        self.obs_sim = torch.from_numpy(tr.obs_sim).cuda()
        self.reuse_in = torch.from_numpy(tr.reuse).cuda()
        b = tr.budget
        self.budget = B.budget_ratio(b.num, b.den) if b.mode == "ratio" else B.budget_count(b.count)
        self.out = {k: B.SelectOutputs.allocate(tr.T, tr.n_steps, tr.T, "cuda") for k in ("static", "ws")}
        self.reuse_out = {k: torch.empty_like(self.reuse_in) for k in ("static", "ws")}
        self.status = {k: B.new_status() for k in ("static", "ws")}

    def steps(self, B, which):
        return B.StepSignals(self.valid, self.gain, self.red, self.reuse_in, self.obs_sim, self.reuse_out[which])

    def run(self, B, which):
        args = (self.sal, self.step_id, self.prot, self.steps(B, which), B.Params(), self.budget, self.out[which])
        if which == "static":
            B.stepkv_select_static_scratch(*args, status=self.status[which])
        else:
            B.stepkv_select(*args, status=self.status[which])

    def compare(self):
        s, w = self.out["static"], self.out["ws"]
        assert int(self.status["static"].item()) == 0 and int(self.status["ws"].item()) == 0
        n = int(w.n_kept.item())
        assert int(s.n_kept.item()) == n
        assert np.array_equal(s.n_budget.cpu().numpy(), w.n_budget.cpu().numpy())
        assert np.array_equal(s.kept_idx[:n].cpu().numpy(), w.kept_idx[:n].cpu().numpy())
        for name in ("step_count", "step_kept"):
            assert np.array_equal(getattr(s, name).cpu().numpy(), getattr(w, name).cpu().numpy()), name
        for name in ("priority", "token_sal", "step_util", "step_sal_sum", "step_sal_max"):
            _assert_close(getattr(s, name).cpu().numpy(), getattr(w, name).cpu().numpy(), name)
        _assert_close(self.reuse_out["static"].cpu().numpy(), self.reuse_out["ws"].cpu().numpy(), "reuse_out")

    def compare_oracle(self):
        """The static-scratch outputs against the CPU oracle on the same saliency rows (T_i = mean of the
        three rows, then Eqs. 1-5 and Algorithm 1)."""
        from oracle import stepkv_oracle as O
        tr, o = self.tr, self.out["static"]
        b = tr.budget
        ref = O.stepkv_boundary([self.sal.cpu().numpy().astype(np.float64)], tr.step_id, tr.prot, tr.valid, tr.gain,
                                tr.red, tr.obs_sim, tr.reuse, O.Params(), b.mode, b.num, b.den, b.count)
        n = int(o.n_kept.item())
        assert n == len(ref["kept"])
        assert TL.compare_kept(o.kept_idx[:n].cpu().numpy().astype(np.int64), ref) == 0
        prunable = ~tr.prot.astype(bool)
        TL.assert_close(o.priority.cpu().numpy()[prunable], ref["P"][prunable], "P vs oracle", floor=1e-6)
        TL.assert_close(o.step_util.cpu().numpy(), ref["S"], "S_k vs oracle", floor=1e-6)
        TL.assert_close(self.reuse_out["static"].cpu().numpy(), ref["reuse"], "c_k vs oracle", floor=1e-6)
        assert np.array_equal(o.step_count.cpu().numpy(), ref["step_count"])
        assert np.array_equal(o.step_kept.cpu().numpy(), ref["step_kept"])
        TL.assert_close(o.step_sal_sum.cpu().numpy(), ref["step_sal_sum"], "step_sal_sum vs oracle", floor=1e-9)
        TL.assert_close(o.step_sal_max.cpu().numpy(), ref["step_sal_max"], "step_sal_max vs oracle", floor=1e-9)


def test_static_scratch_matches_workspace_entry_point_twice_in_a_row(B):
    """Two static-scratch calls back to back on one stream (a cluster-sized trajectory, then a
    single-CTA one with other step counts), each against stepkv_select on the same inputs."""
    import torch
    cases = [
        _Case(B, wl.custom(41, L=1, Hq=4, Hkv=1, d=64, T=20000, W=64, n_steps=40, budget=wl.Budget.ratio(1, 10)), 1),
        _Case(B, wl.custom(42, L=1, Hq=4, Hkv=1, d=64, T=1900, W=16, n_steps=9, budget=wl.Budget.fixed(300)), 2),
    ]
    for c in cases:
        c.run(B, "static")
    for c in cases:
        c.run(B, "ws")
    torch.cuda.synchronize()
    for c in cases:
        c.compare()
        c.compare_oracle()


def test_static_scratch_call_allocates_nothing(B):
    """After the first call on the device (the set-up), a call leaves torch's allocator untouched and
    the device's free memory (cudaMemGetInfo) unchanged: nothing inside the library allocates either."""
    import torch
    c = _Case(B, wl.custom(43, L=1, Hq=4, Hkv=1, d=64, T=7000, W=32, n_steps=12, budget=wl.Budget.ratio(1, 5)), 3)
    c.run(B, "static")
    torch.cuda.synchronize()
    alloc, reserved = torch.cuda.memory_allocated(), torch.cuda.memory_reserved()
    free0, _ = torch.cuda.mem_get_info()
    c.run(B, "static")
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert torch.cuda.memory_allocated() == alloc and torch.cuda.memory_reserved() == reserved
    assert free1 == free0, (free0, free1)
    c.run(B, "ws")
    torch.cuda.synchronize()
    c.compare()


def test_static_scratch_rejects_sizes_above_its_limit(B):
    """n_steps above the scratch limit: STEPKV_ENOSPACE from the C entry point before anything runs,
    and a ValueError from the binding."""
    import torch
    n_steps = B.STATIC_SCRATCH_MAX_STEPS + 1
    tr = wl.custom(44, L=1, Hq=4, Hkv=1, d=64, T=20000, W=16, n_steps=n_steps, budget=wl.Budget.ratio(1, 10))
    c = _Case(B, tr, 4)
    with pytest.raises(ValueError, match="static scratch"):
        c.run(B, "static")
    lib = B.load_library()
    o = c.out["static"]
    o.n_kept.fill_(-5)
    cs, cp, co = c.steps(B, "static").c(), B.Params().c(), o.c()
    code = lib.stepkv_select_static_scratch(c.sal.data_ptr(), 3, tr.T, c.step_id.data_ptr(), c.prot.data_ptr(),
                                            ctypes.byref(cs), ctypes.byref(cp), ctypes.byref(c.budget),
                                            ctypes.byref(co), c.status["static"].data_ptr(),
                                            torch.cuda.current_stream().cuda_stream)
    assert code == B.STEPKV_ENOSPACE
    torch.cuda.synchronize()
    assert int(o.n_kept.item()) == -5 and int(c.status["static"].item()) == 0
    # the workspace entry point takes the same problem
    c.run(B, "ws")
    torch.cuda.synchronize()
    assert int(c.status["ws"].item()) == 0 and int(c.out["ws"].n_kept.item()) > 0
