"""Helpers shared by the parity tests: move generated inputs to the GPU, run the library through the
C ABI binding, run the CPU oracle on the same inputs, and compare under the parity rules:

* floating point (saliency, step scores, priorities, step sums): max relative error <= 2e-3,
  |gpu - oracle| <= 2e-3 * |oracle| (fp32 accumulation from bf16 inputs vs fp64);
* retained sets: bit-exact except swaps in which every differing token's oracle priority lies
  within 2e-3 * |P_B| of the oracle's B-th priority P_B (counted);
* compacted K/V, step ids, positions: bit-exact.
"""
from __future__ import annotations

import numpy as np

from oracle import stepkv_oracle as O
from paper_2609_22158_gb300 import workload as wl

RTOL = 2e-3


def torch():
    import torch as _t
    return _t


def bf16_dev(bits: np.ndarray):
    t = torch()
    return t.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(t.bfloat16).cuda()


def bits_of(x) -> np.ndarray:
    return x.view(torch().int16).cpu().numpy().view(np.uint16)


def oracle_params(p) -> "O.Params":
    return O.Params(lam=p.lam, w_r=p.w_r, w_c=p.w_c, r_min=p.r_min, r_max=p.r_max, s_max=p.s_max, eta=p.eta,
                    alpha=p.alpha, beta=p.beta, sal_norm="max" if p.sal_norm == 0 else "none",
                    pool=getattr(p, "sal_pool", 1), pool_mode="max" if getattr(p, "sal_pool_mode", 0) == 0 else "avg")


def max_rel_err(g, o, floor: float = 0.0) -> float:
    g = np.asarray(g, np.float64)
    o = np.asarray(o, np.float64)
    den = np.maximum(np.abs(o), floor)
    with np.errstate(divide="ignore", invalid="ignore"):
        e = np.where(den > 0, np.abs(g - o) / den, np.abs(g - o))
    return float(e.max()) if e.size else 0.0


def assert_close(g, o, what: str, rtol: float = RTOL, floor: float = 0.0):
    e = max_rel_err(g, o, floor)
    assert e <= rtol, f"{what}: max relative error {e:.3e} > {rtol}"
    return e


# Decode outputs are weighted sums out_e = sum_j p_j V[j, e] whose terms cancel: a float sum's rounding
# error is bounded relative to the magnitude of its terms, m_e = sum_j p_j |V[j, e]|, not to |out_e|.  The
# element-wise rule is therefore |g - o| <= RTOL * max(|o_e|, DECODE_FLOOR * m_e): the 2e-3 relative
# rule in full wherever the cancellation is below 1000x, and 2e-6 of the terms' magnitude beyond.
DECODE_FLOOR = 1e-3


def assert_decode_close(g, q_bits, K_bits, V_bits, what: str):
    """Element-wise decode parity against the oracle (see DECODE_FLOOR); returns the max relative error."""
    o = O.decode_attention(q_bits, K_bits, V_bits)
    m = O.decode_attention(q_bits, K_bits, np.asarray(V_bits, np.uint16) & np.uint16(0x7FFF))  # |V|
    g = np.asarray(g, np.float64)
    den = np.maximum(np.abs(o), DECODE_FLOOR * m)
    e = np.abs(g - o) / den
    worst = np.unravel_index(int(np.argmax(e)), e.shape)
    assert e.max() <= RTOL, (f"{what}: element {worst}: gpu {g[worst]:.6e} oracle {o[worst]:.6e} "
                             f"(terms' magnitude {m[worst]:.3e}), relative error {e.max():.3e} > {RTOL}")
    return float(e.max())


def compare_kept(gpu_kept: np.ndarray, out: dict, rtol: float = RTOL) -> int:
    """Retained-set rule; returns the number of tolerated swaps."""
    o_kept = out["kept"]
    if np.array_equal(gpu_kept, o_kept):
        return 0
    assert len(gpu_kept) == len(o_kept), f"retained count {len(gpu_kept)} != oracle {len(o_kept)}"
    assert np.all(np.diff(gpu_kept) > 0), "retained slots not strictly ascending"
    diff = np.setxor1d(gpu_kept, o_kept)
    P = out["P"]
    chosen = out["chosen"]
    PB = np.sort(P[chosen])[0] if len(chosen) else 0.0
    tol = rtol * abs(PB)
    bad = [int(i) for i in diff if not (np.isfinite(P[i]) and abs(P[i] - PB) <= tol)]
    assert not bad, f"retained sets differ beyond tolerance at slots {bad[:10]} (P_B={PB})"
    return len(diff) // 2


class GpuTraj:
    """A workload trajectory materialised on the GPU (all layers)."""

    def __init__(self, tr: "wl.Trajectory", layers=None, kept_cap=None, params=None):
        t = torch()
        self.tr = tr
        s = tr.shape
        self.L = s.L
        self.K = [bf16_dev(tr.keys(l)) for l in range(s.L)]
        self.V = [bf16_dev(tr.values(l)) for l in range(s.L)]
        self.Q = [bf16_dev(tr.queries(l)) for l in tr.sal_layer_ids()]
        self.step_id = t.from_numpy(tr.step_id).cuda()
        self.prot = t.from_numpy(tr.prot).cuda()
        self.pos = t.from_numpy(tr.pos).cuda()
        self.valid = t.from_numpy(tr.valid).cuda()
        self.gain = t.from_numpy(tr.gain).cuda()
        self.red = t.from_numpy(tr.red).cuda()
        self.obs_sim = t.from_numpy(tr.obs_sim).cuda()
        self.reuse_in = t.from_numpy(tr.reuse).cuda()
        self.reuse_out = t.empty_like(self.reuse_in)
        n_prot = int(tr.prot.sum())
        self.kept_cap = kept_cap if kept_cap is not None else s.T
        self.n_prot = n_prot

    def budget(self):
        from paper_2609_22158_gb300 import binding as B
        b = self.tr.budget
        return B.budget_ratio(b.num, b.den) if b.mode == "ratio" else B.budget_count(b.count)

    def steps(self):
        from paper_2609_22158_gb300 import binding as B
        return B.StepSignals(self.valid, self.gain, self.red, self.reuse_in, self.obs_sim, self.reuse_out)

    def problem(self, budget=None):
        t = torch()
        from paper_2609_22158_gb300 import binding as B
        s = self.tr.shape
        cap = self.kept_cap
        self.K_out = [t.empty((s.Hkv, cap, s.d), dtype=t.bfloat16, device="cuda") for _ in range(s.L)]
        self.V_out = [t.empty((s.Hkv, cap, s.d), dtype=t.bfloat16, device="cuda") for _ in range(s.L)]
        self.out = B.SelectOutputs.allocate(s.T, self.tr.n_steps, cap, "cuda")
        self.step_id_out = t.full((cap,), -7, dtype=t.int32, device="cuda")
        self.pos_out = t.full((cap,), -7, dtype=t.int32, device="cuda")
        return B.Problem(self.K, self.V, self.Q, s.T, self.step_id, self.prot, self.steps(),
                         budget if budget is not None else self.budget(),
                         self.K_out, self.V_out, self.out, pos_in=self.pos, step_id_out=self.step_id_out,
                         pos_out=self.pos_out)


def run_oracle(tr: "wl.Trajectory", p: "O.Params") -> dict:
    Ks = [tr.keys(l) for l in tr.sal_layer_ids()]
    Qs = [tr.queries(l) for l in tr.sal_layer_ids()]
    b = tr.budget
    return O.compress(Ks, Qs, tr.step_id, tr.prot, tr.valid, tr.gain, tr.red, tr.obs_sim, tr.reuse, p, b.mode, b.num,
                      b.den, b.count)


def check_select_outputs(g: GpuTraj, out: dict, n_kept_expected=None) -> int:
    """Compare every selection output of the library against the oracle dict; returns swaps."""
    o = g.out
    tr = g.tr
    n_kept = int(o.n_kept.item())
    gk = o.kept_idx[:n_kept].cpu().numpy().astype(np.int64)
    nb = o.n_budget.cpu().numpy()
    assert nb[0] == out["N"] and nb[1] == out["B"], (nb, out["N"], out["B"])
    assert n_kept == len(out["kept"]), (n_kept, len(out["kept"]))
    prunable = ~tr.prot.astype(bool)
    assert_close(o.step_util.cpu().numpy(), out["S"], "S_k", floor=1e-6)
    assert_close(g.reuse_out.cpu().numpy(), out["reuse"], "c_k", floor=1e-6)
    assert_close(o.token_sal.cpu().numpy()[prunable], out["T_hat"][prunable], "T_hat")
    Pg = o.priority.cpu().numpy()
    assert np.all(np.isneginf(Pg[~prunable]))
    assert_close(Pg[prunable], out["P"][prunable], "P", floor=1e-6)
    assert np.array_equal(o.step_count.cpu().numpy(), out["step_count"])
    assert_close(o.step_sal_sum.cpu().numpy(), out["step_sal_sum"], "step_sal_sum", floor=1e-9)
    assert_close(o.step_sal_max.cpu().numpy(), out["step_sal_max"], "step_sal_max", floor=1e-9)
    swaps = compare_kept(gk, out)
    sk = o.step_kept.cpu().numpy()
    if swaps == 0:
        assert np.array_equal(sk, out["step_kept"])
    assert sk.sum() == out["B"]
    return swaps
