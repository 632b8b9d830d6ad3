"""Seeded synthetic agent-trajectory workloads.

This module only draws random inputs: KV caches, window queries, the layout of
reasoning steps over the token axis and the per-step trajectory signals.  It
holds none of StepKV's arithmetic (no saliency, no utility, no selection), so
both the CUDA path and the CPU oracle can be fed from it.

Conventions (the paper's notation, Sec. 3 "Problem Formulation"):

* a trajectory is the prompt followed by steps k = 0..t-1 (0-based here), each
  step a contiguous span Thought || Action || Observation that shares one step
  id (Sec. 3: "each completed step occupies a contiguous span");
* the first ``n_prompt`` slots are the protected prompt/query tokens
  (step id -1) and the last ``W`` slots are the observation window, also
  protected, lying at the end of the last step;
* K/V per layer are ``[Hkv, T, d]`` bf16, window queries ``[Hq, W, d]`` bf16,
  both stored here as raw ``uint16`` bf16 bit patterns (round-to-nearest-even
  from fp32 N(0, 1) draws).

Random streams: one ``numpy.random.PCG64`` per array, spawned from one
``SeedSequence(seed)`` by a fixed key, so every array is reproducible on its
own and a trajectory can be regenerated lazily layer by layer.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional, Sequence, Tuple

import numpy as np

FIELD_PROMPT, FIELD_THOUGHT, FIELD_ACTION, FIELD_OBSERVATION = 0, 1, 2, 3

# Table H defaults are not needed here: this module draws inputs only.


def _rng(seed: int, *key: int) -> np.random.Generator:
    """Independent PCG64 stream for (seed, key...)."""
    ss = np.random.SeedSequence([int(seed) & 0xFFFFFFFF] + [int(k) & 0xFFFFFFFF for k in key])
    return np.random.Generator(np.random.PCG64(ss))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit patterns, round to nearest even (inputs are finite)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = u + (np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1)))
    return (rounded >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


# Stream keys (stable: changing one changes the workload).
_K_LAYOUT, _K_SIGNALS, _K_KEYS, _K_VALUES, _K_QUERIES, _K_NEEDLE, _K_OUTLIER = 1, 2, 3, 4, 5, 6, 7


@dataclass
class Budget:
    """KV budget: a keep ratio rho = num/den of the prunable count (Eq. 1), or a fixed count."""
    mode: str = "ratio"  # "ratio" | "count"
    num: int = 1
    den: int = 10
    count: int = 0

    @staticmethod
    def ratio(num: int, den: int) -> "Budget":
        return Budget("ratio", int(num), int(den), 0)

    @staticmethod
    def fixed(count: int) -> "Budget":
        return Budget("count", 0, 1, int(count))


@dataclass
class Shape:
    L: int
    Hq: int
    Hkv: int
    d: int
    T: int
    W: int
    n_sal_layers: int = 3

    @property
    def G(self) -> int:
        return self.Hq // self.Hkv

    @property
    def Ls(self) -> int:
        return min(self.n_sal_layers, self.L)


@dataclass
class Trajectory:
    """One agent trajectory at a pruning boundary (after step t = n_steps-1)."""
    name: str
    seed: int
    shape: Shape
    n_prompt: int
    step_id: np.ndarray      # int32 [T], -1 for the prompt
    field: np.ndarray        # int8  [T], FIELD_*
    prot: np.ndarray         # uint8 [T], 1 = protected (prompt + window)
    pos: np.ndarray          # int32 [T], original positions
    valid: np.ndarray        # float32 [n_steps]  valid_k in {0,1}
    gain: np.ndarray         # float32 [n_steps]  gain_k in [0,1]
    red: np.ndarray          # float32 [n_steps]  red_k in [0,1]
    obs_sim: np.ndarray      # float32 [n_steps]  sim(Obs_t, Obs_k)
    reuse: np.ndarray        # float32 [n_steps]  c_k before this boundary
    budget: Budget
    needles: List[Tuple[int, int]] = field(default_factory=list)  # (start, length)
    outlier_scale: float = 1.0
    outlier_channels: int = 0
    kv_std: float = 1.0

    @property
    def n_steps(self) -> int:
        return int(self.valid.shape[0])

    @property
    def T(self) -> int:
        return self.shape.T

    # ---- lazily generated tensors (bf16 bits) ----
    def sal_layer_ids(self) -> List[int]:
        s = self.shape
        return list(range(s.L - s.Ls, s.L))

    def queries(self, layer: int) -> np.ndarray:
        """Window queries of one layer, [Hq, W, d] bf16 bits."""
        s = self.shape
        g = _rng(self.seed, _K_QUERIES, layer)
        q = g.standard_normal((s.Hq, s.W, s.d), dtype=np.float32)
        return f32_to_bf16_bits(q)

    def keys(self, layer: int) -> np.ndarray:
        """K of one layer, [Hkv, T, d] bf16 bits (needles and outlier channels planted)."""
        s = self.shape
        g = _rng(self.seed, _K_KEYS, layer)
        k = g.standard_normal((s.Hkv, s.T, s.d), dtype=np.float32)
        if self.kv_std != 1.0:
            k *= np.float32(self.kv_std)
        if self.needles:
            q = bf16_bits_to_f32(self.queries(layer)).reshape(s.Hkv, s.G * s.W, s.d)
            gn = _rng(self.seed, _K_NEEDLE, layer)
            for h in range(s.Hkv):
                u = q[h].astype(np.float64).mean(axis=0)
                u /= np.linalg.norm(u)
                for (st, ln) in self.needles:
                    z = gn.standard_normal((ln, s.d))
                    z -= np.outer(z @ u, u)
                    z /= np.linalg.norm(z, axis=1, keepdims=True)
                    k[h, st:st + ln] = (np.sqrt(s.d) * (0.3 * u[None, :] + np.sqrt(0.91) * z)).astype(np.float32)
        if self.outlier_channels > 0:
            go = _rng(self.seed, _K_OUTLIER, layer)
            for h in range(s.Hkv):
                ch = go.choice(s.d, size=self.outlier_channels, replace=False)
                k[h][:, ch] *= np.float32(self.outlier_scale)
        return f32_to_bf16_bits(k)

    def values(self, layer: int) -> np.ndarray:
        s = self.shape
        g = _rng(self.seed, _K_VALUES, layer)
        return f32_to_bf16_bits(g.standard_normal((s.Hkv, s.T, s.d), dtype=np.float32))


def _rescale_lengths(lens: np.ndarray, total: int) -> np.ndarray:
    """Scale positive integer lengths to sum exactly to `total`, each >= 1 (largest remainder)."""
    lens = np.asarray(lens, dtype=np.float64).ravel()
    n = lens.size
    if total < n:
        raise ValueError("total smaller than the number of fields")
    scaled = lens * (total / lens.sum())
    base = np.maximum(np.floor(scaled).astype(np.int64), 1)
    rem = total - int(base.sum())
    frac = scaled - np.floor(scaled)
    if rem > 0:
        order = np.argsort(-frac, kind="stable")
        for i in range(rem):
            base[order[i % n]] += 1
    elif rem < 0:
        order = np.argsort(-base, kind="stable")
        i = 0
        while rem < 0:
            j = order[i % n]
            if base[j] > 1:
                base[j] -= 1
                rem += 1
            i += 1
    assert int(base.sum()) == total and base.min() >= 1
    return base


def _assemble(name, seed, shape, n_prompt, field_lens, budget, g_sig, needles_steps=0, **kw) -> Trajectory:
    """field_lens: int [n_steps, 3] (Th, Act, Obs) lengths summing to T - n_prompt."""
    T = shape.T
    n_steps = field_lens.shape[0]
    step_id = np.full(T, -1, dtype=np.int32)
    fld = np.zeros(T, dtype=np.int8)
    pos = n_prompt
    obs_spans = []
    for k in range(n_steps):
        for f in range(3):
            ln = int(field_lens[k, f])
            step_id[pos:pos + ln] = k
            fld[pos:pos + ln] = f + 1
            if f == 2:
                obs_spans.append((pos, ln))
            pos += ln
    assert pos == T
    prot = np.zeros(T, dtype=np.uint8)
    prot[:n_prompt] = 1
    prot[T - shape.W:] = 1
    valid = (g_sig.random(n_steps) >= 0.2).astype(np.float32)
    gain = g_sig.random(n_steps).astype(np.float32)
    red = g_sig.random(n_steps).astype(np.float32)
    obs_sim = g_sig.random(n_steps).astype(np.float32)
    # prior reuse accumulators: any value in [0, number of earlier boundaries that could have credited step k]
    t = n_steps - 1
    reuse = (g_sig.random(n_steps) * np.maximum(t - 1 - np.arange(n_steps), 0)).astype(np.float32)
    reuse[t] = np.float32(0.5)  # stale value: the current step's accumulator must be reset to zero
    needles = []
    if needles_steps:
        g_n = _rng(seed, _K_NEEDLE, 10_000)
        cand = [s for s in obs_spans[1:1 + needles_steps] if s[1] >= 16]
        for (st, ln) in cand[:3]:
            off = int(g_n.integers(0, ln - 16 + 1))
            needles.append((st + off, 16))
    traj = Trajectory(name=name, seed=seed, shape=shape, n_prompt=n_prompt, step_id=step_id, field=fld, prot=prot,
                      pos=np.arange(T, dtype=np.int32), valid=valid, gain=gain, red=red, obs_sim=obs_sim,
                      reuse=reuse, budget=budget, needles=needles, **kw)
    return traj


def _cycle_steps(g, n_steps, th, act, obs, total, W, obs_log=False) -> np.ndarray:
    for _ in range(1000):
        lens = np.empty((n_steps, 3), dtype=np.int64)
        lens[:, 0] = g.integers(th[0], th[1] + 1, n_steps)
        lens[:, 1] = g.integers(act[0], act[1] + 1, n_steps)
        if obs_log:
            lens[:, 2] = np.round(np.exp(g.uniform(np.log(obs[0]), np.log(obs[1]), n_steps))).astype(np.int64)
        else:
            lens[:, 2] = g.integers(obs[0], obs[1] + 1, n_steps)
        out = _rescale_lengths(lens, total).reshape(n_steps, 3)
        if out[-1].sum() >= W + 1:
            return out
    raise RuntimeError("could not draw a step layout with a last step longer than the window")


def tiny(seed: int = 0, budget: Optional[Budget] = None) -> Trajectory:
    """1 layer, Hq=8/Hkv=2 (GQA 4), d=64, T=2048, W=32, 8 steps of U{100..400} tokens
    (last step absorbs the remainder), prompt 16, budget 25% of the prunable tokens."""
    shape = Shape(L=1, Hq=8, Hkv=2, d=64, T=2048, W=32)
    g = _rng(seed, _K_LAYOUT)
    n_prompt, total = 16, 2048 - 16
    for _ in range(1000):
        lens = g.integers(100, 401, 7)
        last = total - int(lens.sum())
        if last >= shape.W + 1 + 3:
            break
    step_lens = np.append(lens, last)
    fl = np.empty((8, 3), dtype=np.int64)
    for k, sl in enumerate(step_lens):
        parts = np.array([g.integers(50, 301), g.integers(10, 51), g.integers(200, 2001)])
        fl[k] = _rescale_lengths(parts, int(sl))
    return _assemble("tiny", seed, shape, n_prompt, fl, budget or Budget.ratio(1, 4), _rng(seed, _K_SIGNALS))


def llama8b_32k(seed: int = 1, budget: Optional[Budget] = None, T: int = 32768, L: int = 32,
                n_steps: int = 40, needles: bool = True, W: int = 64) -> Trajectory:
    """Llama-3-8B-shaped single trajectory: L=32, Hq=32/Hkv=8, d=128, T=32768, 40 steps cycling
    Thought (50-300) / Action (10-50) / Observation (200-2000), rescaled to fill the context;
    3 needle spans of 16 keys in early Observations aligned with the window queries (cos ~0.3);
    window 64; budget 10%."""
    shape = Shape(L=L, Hq=32, Hkv=8, d=128, T=T, W=W)
    g = _rng(seed, _K_LAYOUT)
    fl = _cycle_steps(g, n_steps, (50, 300), (10, 50), (200, 2000), T - 16, W)
    return _assemble("llama8b_32k", seed, shape, 16, fl, budget or Budget.ratio(1, 10), _rng(seed, _K_SIGNALS),
                     needles_steps=5 if needles else 0)


def observation_prefill(base: str = "llama8b_32k", W: int = 2048, seed: Optional[int] = None,
                        budget: Optional[Budget] = None) -> Trajectory:
    """Saliency from the whole last Observation instead of a short window: the queries are the |Obs_t| = W
    tokens of the step just completed (the appendix's time-complexity passage collects T_i during the
    observation prefill).  The layout is the base workload's (Llama-3-8B 32K: 40 steps, 10%; Qwen2.5-32B
    64K: 120 steps, log-uniform Observations, 4096 tokens), except that the last step's Observation is
    exactly W tokens long and is the protected window."""
    if base == "llama8b_32k":
        seed = 1 if seed is None else seed
        shape = Shape(L=32, Hq=32, Hkv=8, d=128, T=32768, W=W)
        n_steps, obs, obs_log, nd = 40, (200, 2000), False, 5
        budget = budget or Budget.ratio(1, 10)
    elif base == "qwen32b_64k":
        seed = 3 if seed is None else seed
        shape = Shape(L=64, Hq=40, Hkv=8, d=128, T=65536, W=W)
        n_steps, obs, obs_log, nd = 120, (16, 4096), True, 0
        budget = budget or Budget.fixed(4096)
    else:
        raise ValueError(base)
    g = _rng(seed, _K_LAYOUT, 20_000 + W)
    fl = _cycle_steps(g, n_steps, (50, 300), (10, 50), obs, shape.T - 16 - W, 0, obs_log=obs_log)
    fl[-2, 2] += fl[-1, 2]  # the drawn last Observation joins the previous one; the last is exactly W
    fl[-1, 2] = W
    return _assemble(f"{base}_obs{W}", seed, shape, 16, fl, budget, _rng(seed, _K_SIGNALS), needles_steps=nd)


def ragged_batch(seed: int = 2, n_traj: int = 16, budget: Optional[Budget] = None, L: int = 32,
                 t_lo: int = 8192, t_hi: int = 32768) -> List[Trajectory]:
    """16 trajectories, T ~ U(8K, 32K), Llama-3-8B head shapes, 24-60 steps each, 4 key channels
    per (layer, KV head) scaled x8 before bf16 rounding, window 64."""
    g = _rng(seed, _K_LAYOUT, 999)
    out = []
    for b in range(n_traj):
        T = int(g.integers(t_lo, t_hi + 1))
        n_steps = int(g.integers(24, 61))
        shape = Shape(L=L, Hq=32, Hkv=8, d=128, T=T, W=64)
        sub = seed * 1000 + 17 + b
        gl = _rng(sub, _K_LAYOUT)
        fl = _cycle_steps(gl, n_steps, (50, 300), (10, 50), (200, 2000), T - 16, 64)
        out.append(_assemble(f"ragged{b}", sub, shape, 16, fl, budget or Budget.ratio(1, 10), _rng(sub, _K_SIGNALS),
                             outlier_scale=8.0, outlier_channels=4))
    return out


def qwen32b_64k(seed: int = 3, budget: Optional[Budget] = None, T: int = 65536, L: int = 64) -> Trajectory:
    """Qwen2.5-32B-shaped long horizon: L=64, Hq=40/Hkv=8, d=128, T=65536, 120 steps,
    Observations log-uniform in [16, 4096] tokens before rescaling, window 128, fixed budget 4096."""
    shape = Shape(L=L, Hq=40, Hkv=8, d=128, T=T, W=128)
    g = _rng(seed, _K_LAYOUT)
    fl = _cycle_steps(g, 120, (50, 300), (10, 50), (16, 4096), T - 16, 128, obs_log=True)
    return _assemble("qwen32b_64k", seed, shape, 16, fl, budget or Budget.fixed(4096), _rng(seed, _K_SIGNALS))


def custom(seed: int, L: int, Hq: int, Hkv: int, d: int, T: int, W: int, n_steps: int, n_prompt: int = 16,
           budget: Optional[Budget] = None, n_sal_layers: int = 3, outlier_channels: int = 0,
           kv_std: float = 1.0) -> Trajectory:
    """Arbitrary small shape for parity and edge-case tests (steps cycle the Llama field ranges)."""
    shape = Shape(L=L, Hq=Hq, Hkv=Hkv, d=d, T=T, W=W, n_sal_layers=n_sal_layers)
    g = _rng(seed, _K_LAYOUT)
    total = T - n_prompt
    if n_steps * 3 > total:
        raise ValueError("too many steps for T")
    for _ in range(1000):
        lens = np.empty((n_steps, 3), dtype=np.int64)
        lens[:, 0] = g.integers(50, 301, n_steps)
        lens[:, 1] = g.integers(10, 51, n_steps)
        lens[:, 2] = g.integers(200, 2001, n_steps)
        fl = _rescale_lengths(lens, total).reshape(n_steps, 3)
        if fl[-1].sum() >= min(W, total - 3 * (n_steps - 1)):
            break
    return _assemble(f"custom{T}", seed, shape, n_prompt, fl, budget or Budget.ratio(1, 5), _rng(seed, _K_SIGNALS),
                     outlier_scale=8.0, outlier_channels=outlier_channels, kv_std=kv_std)


class IncrementalLoop:
    """The incremental agent loop: a trajectory that grows by one step per boundary.  After every step,
    the already-compacted cache plus the new step is compressed again under a fixed budget, and the
    agent then decodes over the compacted cache.

    This class draws only the new material of each boundary: the rows of the new step (K/V per layer,
    step id, original positions), the window queries, and the per-step signals.  The compacted state
    (retained rows, their step ids and positions, the reuse accumulators) is carried by the caller from
    one boundary to the next.  The first boundary compresses an initial trajectory of ``t0`` tokens
    (prompt + steps); every later boundary adds one step with the config-2 field ranges, the Observation
    at least W + 1 tokens long so that the window lies inside the new step.
    """

    def __init__(self, seed: int, L: int, Hq: int, Hkv: int, d: int, W: int, t0: int, budget_count: int,
                 n_prompt: int = 16, n_steps0: int = 8, n_sal_layers: int = 3, n_boundaries=None,
                 growth_total=None):
        self.seed = int(seed)
        self.shape = Shape(L=L, Hq=Hq, Hkv=Hkv, d=d, T=t0, W=W, n_sal_layers=n_sal_layers)
        self.t0 = int(t0)
        self.n_prompt = int(n_prompt)
        self.budget = Budget.fixed(budget_count)
        g = _rng(seed, _K_LAYOUT, 50_000)
        self.init_fields = _cycle_steps(g, n_steps0, (50, 300), (10, 50), (200, 2000), t0 - n_prompt, W)
        # With growth_total, the steps of boundaries 1 .. n_boundaries-1 are drawn as below and then
        # rescaled (largest remainder) to add exactly growth_total tokens over the loop, e.g. 200
        # boundaries growing a 4096-token start to 131072 tokens (mean ~635 tokens per step).
        self._scaled = None
        if growth_total is not None:
            raw = np.array([self._raw_step_length(b) for b in range(1, int(n_boundaries))], dtype=np.int64)
            self._scaled = _rescale_lengths(raw, int(growth_total))
            if self._scaled.min() < W + 1:
                raise ValueError("rescaled steps shorter than the window")

    # ---- layout
    def _raw_step_length(self, b: int) -> int:
        g = _rng(self.seed, _K_LAYOUT, 60_000 + b)
        th, act = int(g.integers(50, 301)), int(g.integers(10, 51))
        obs = max(int(g.integers(200, 2001)), self.shape.W + 1)
        return th + act + obs

    def step_length(self, b: int) -> int:
        """Tokens of the step added at boundary b >= 1 (Thought + Action + Observation)."""
        if self._scaled is not None:
            return int(self._scaled[b - 1])
        return self._raw_step_length(b)

    def initial_layout(self):
        """(step_id [t0], n_steps) of the first boundary's trajectory."""
        step_id = np.full(self.t0, -1, dtype=np.int32)
        pos = self.n_prompt
        for k, row in enumerate(self.init_fields):
            ln = int(row.sum())
            step_id[pos:pos + ln] = k
            pos += ln
        return step_id, int(self.init_fields.shape[0])

    # ---- rows (bf16 bits)
    def rows(self, b: int, layer: int, which: int, n: int) -> np.ndarray:
        """New rows of boundary b for one layer: [Hkv, n, d]; which = _K_KEYS or _K_VALUES.  Boundary 0's
        rows are the initial trajectory."""
        s = self.shape
        g = _rng(self.seed, which, layer, 70_000 + b)
        return f32_to_bf16_bits(g.standard_normal((s.Hkv, n, s.d), dtype=np.float32))

    def queries(self, b: int, layer: int) -> np.ndarray:
        """Window queries of boundary b, [Hq, W, d]."""
        s = self.shape
        g = _rng(self.seed, _K_QUERIES, layer, 80_000 + b)
        return f32_to_bf16_bits(g.standard_normal((s.Hq, s.W, s.d), dtype=np.float32))

    # ---- signals
    def signals(self, b: int, n_steps: int):
        """valid/gain/red of steps 0..n_steps-1 (fixed once drawn per step) and this boundary's obs_sim."""
        valid = np.empty(n_steps, np.float32)
        gain = np.empty(n_steps, np.float32)
        red = np.empty(n_steps, np.float32)
        for k in range(n_steps):
            g = _rng(self.seed, _K_SIGNALS, 90_000 + k)
            valid[k] = np.float32(g.random() >= 0.2)
            gain[k] = np.float32(g.random())
            red[k] = np.float32(g.random())
        obs_sim = _rng(self.seed, _K_SIGNALS, 95_000 + b).random(n_steps).astype(np.float32)
        return valid, gain, red, obs_sim

    def protected(self, step_id: np.ndarray) -> np.ndarray:
        """Prompt rows (step id -1) and the last W rows (the window of the newest step)."""
        prot = (step_id < 0).astype(np.uint8)
        prot[-self.shape.W:] = 1
        return prot


def decode_queries(seed: int, n_layers: int, Hq: int, d: int, n: int) -> np.ndarray:
    """Single-token decode queries [n, n_layers, Hq, d] bf16 bits."""
    g = _rng(seed, _K_QUERIES, 77_777)
    return f32_to_bf16_bits(g.standard_normal((n, n_layers, Hq, d), dtype=np.float32))


def synthetic_cues(seed: int, n_steps: int, vocab: int = 4000, reuse: float = 0.3, repeat_action: float = 0.25):
    """Evidence cues of every step's fields (Thought, Action, Observation) for the Sec. 4.1 signals: each
    field draws 8-64 distinct ids from a vocabulary; a fraction ``reuse`` of an Observation's and Thought's
    cues repeats cues of a random earlier Observation (later steps reusing earlier evidence), and with
    probability ``repeat_action`` an Action repeats an earlier Action's cues (a redundant tool call).
    Returns [(th, act, obs)] of sorted uint32 arrays."""
    g = _rng(seed, _K_SIGNALS, 123_456)
    steps = []
    for k in range(n_steps):
        fields = []
        for f in range(3):
            n = int(g.integers(8, 65))
            if f == 1 and k > 0 and g.random() < repeat_action:
                fields.append(steps[int(g.integers(0, k))][1].copy())
                continue
            own = g.integers(0, vocab, n)
            if f != 1 and k > 0:
                src = steps[int(g.integers(0, k))][2]
                m = min(len(src), int(reuse * n))
                if m:
                    own[:m] = g.choice(src, m, replace=False)
            fields.append(np.unique(own.astype(np.uint32))[:64])
        steps.append(tuple(fields))
    return steps