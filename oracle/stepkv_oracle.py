"""StepKV CPU oracle (fp64) -- TEST INFRASTRUCTURE ONLY.

Plain, slow, obviously-correct restatement of what StepKV's compression pass
computes at one pruning boundary (arXiv 2609.22158).  It shares no code with
the CUDA library and never calls it.  Only ``tests/``, ``__graft_entry__.smoke()``
and ``bench.py``'s CPU-baseline / reference arm may import it; the product path
must never route through it.

Every function names the passage it follows.  Equations are numbered as in the
paper: Eq. 1 (problem / budget, Sec. 3), Eq. 2 (completion score r_k), Eq. 3
(reuse accumulator c_k), Eq. 4 (step utility S_k), Eq. 5 (retention priority
P_i, Sec. 4.2), Algorithm 1 (the three phases per boundary, appendix "StepKV
Pseudocode"), Table H (default hyper-parameters, appendix "Implementation
Details").  Where the paper is silent or ambiguous the reading taken is stated
at the function (the readings are listed together in the design notes).

Precision: all floating point is fp64.  bf16 inputs are widened exactly.

Library primitives used as single steps: ``numpy.matmul`` (the Q.K^T dot
products), ``numpy.exp``/``numpy.log1p``, ``numpy.lexsort`` (the global ranking),
``numpy.lib.stride_tricks.sliding_window_view`` (the pooling windows).
No blocking, fusion or reordering beyond the definitions.

Pinning status (see tests/test_oracle_pins.py): every function below is pinned
against closed forms, invariants, brute force or hand-computed tables; none is
"parity unpinned".
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import Dict, List, Optional, Sequence

import numpy as np


# --------------------------------------------------------------------------------------
# Table H defaults (appendix, "Implementation hyperparameters and default settings")
# --------------------------------------------------------------------------------------
@dataclass
class Params:
    lam: float = 0.3      # lambda, redundancy penalty in r_k (Eq. 2)
    w_r: float = 0.85     # completion weight (Eq. 4)
    w_c: float = 0.15     # reuse weight (Eq. 4)
    r_min: float = -1.0   # inner clip of r_k (Eq. 4)
    r_max: float = 2.0
    s_max: float = 8.0    # outer clip of S_k (Eq. 4)
    eta: float = 1.5      # reuse update scale (Eq. 3)
    alpha: float = 0.2    # token-saliency weight (Eq. 5)
    beta: float = 0.8     # step-utility weight (Eq. 5)
    sal_norm: str = "max"  # "max": T_i / max over prunable tokens (appendix, H_i in [0, H_max]); "none"
    pool: int = 1          # SnapKV-style pooling width k along the token axis (odd; 1 = none)
    pool_mode: str = "max"  # "max" or "avg" pooling


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to float64."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


# --------------------------------------------------------------------------------------
# Stage 1: token saliency T_i (Sec. 4.2; "conventional attention-based saliency",
# collected from the observation-window queries of the last saliency layers)
# --------------------------------------------------------------------------------------
def window_attention_saliency(K: np.ndarray, Q: np.ndarray, row_chunk: int = 256) -> np.ndarray:
    """Per-KV-head saliency of one layer.

    K: [Hkv, T, d] bf16 bits (keys, already position-encoded).
    Q: [Hq, W, d] bf16 bits (the observation-window queries; query w sits at slot T-W+w).
    Returns A: [Hkv, T] float64 with
        A[h, j] = (1/G) * sum_{g in group(h)} sum_{w} softmax_{j' <= p_w}(q_{g,w} . k_{j'} / sqrt(d))[j]
    where group(h) = q heads h*G .. h*G+G-1 (GQA), p_w = T-W+w, and the softmax runs causally over
    every visible key, protected tokens included.
    """
    K = bf16_to_f64(K)
    Q = bf16_to_f64(Q)
    Hkv, T, d = K.shape
    Hq, W, dq = Q.shape
    assert dq == d and Hq % Hkv == 0 and 1 <= W <= T
    G = Hq // Hkv
    scale = 1.0 / math.sqrt(d)
    A = np.zeros((Hkv, T), dtype=np.float64)
    j = np.arange(T)
    for h in range(Hkv):
        rows_q = Q[h * G:(h + 1) * G].reshape(G * W, d)          # row r = g*W + w
        p = T - W + (np.arange(G * W) % W)                         # slot of each query row
        for r0 in range(0, G * W, row_chunk):
            r1 = min(G * W, r0 + row_chunk)
            s = (rows_q[r0:r1] @ K[h].T) * scale                   # [rows, T] logits
            visible = j[None, :] <= p[r0:r1, None]
            s = np.where(visible, s, -np.inf)
            s = s - s.max(axis=1, keepdims=True)
            e = np.where(visible, np.exp(s), 0.0)
            a = e / e.sum(axis=1, keepdims=True)                   # softmax per query row
            A[h] += a.sum(axis=0)
        A[h] /= G                                                  # mean over the GQA group
    return A


def pool_tokens(a: np.ndarray, k: int, mode: str = "max") -> np.ndarray:
    """SnapKV-style pooling of one saliency row along the token axis (Sec. 4.2 names SnapKV as an
    interchangeable T_i estimator; reading: a 1-D pool of odd width k, stride 1, the window
    [i - k//2, i + k//2] clipped to [0, T), so padding never enters a maximum or an average).
    out[i] = max (or mean) of a[j] over the window."""
    a = np.asarray(a, dtype=np.float64)
    h = k // 2
    if h == 0:
        return a.copy()
    fill = -np.inf if mode == "max" else np.nan
    padded = np.concatenate([np.full(h, fill), a, np.full(h, fill)])
    windows = np.lib.stride_tricks.sliding_window_view(padded, 2 * h + 1)  # [T, k], window i centred on i
    return windows.max(axis=1) if mode == "max" else np.nanmean(windows, axis=1)


def window_row_lse(K: np.ndarray, Q: np.ndarray) -> np.ndarray:
    """Natural-log log-sum-exp of every observation query's causal attention row (what a prefill
    attention kernel reports beside its output): lse[g, w] = log sum_{j <= p_w} exp(q_{g,w} . k_j / sqrt(d)),
    p_w = T-W+w, with the query heads mapped to KV heads as in window_attention_saliency.
    K: [Hkv, T, d] and Q: [Hq, W, d] bf16 bits; returns [Hq, W] float64."""
    K = bf16_to_f64(K)
    Q = bf16_to_f64(Q)
    Hkv, T, d = K.shape
    Hq, W, _ = Q.shape
    G = Hq // Hkv
    scale = 1.0 / math.sqrt(d)
    lse = np.empty((Hq, W), dtype=np.float64)
    for g in range(Hq):
        s = (Q[g] @ K[g // G].T) * scale                           # [W, T] logits
        visible = np.arange(T)[None, :] <= (T - W + np.arange(W))[:, None]
        s = np.where(visible, s, -np.inf)
        m = s.max(axis=1, keepdims=True)
        lse[g] = (m + np.log(np.where(visible, np.exp(s - m), 0.0).sum(axis=1, keepdims=True)))[:, 0]
    return lse


def token_saliency(A_layers: Sequence[np.ndarray], pool: int = 1, pool_mode: str = "max") -> np.ndarray:
    """T_i = mean over (saliency layer, KV head) of A[l, h, i]  (reading: mean pooling); with pool > 1
    each (layer, KV head) row is first pooled along the token axis (pool_tokens)."""
    A = np.stack([np.asarray(a, dtype=np.float64) for a in A_layers])  # [Ls, Hkv, T]
    if pool > 1:
        A = np.stack([[pool_tokens(row, pool, pool_mode) for row in layer] for layer in A])
    return A.mean(axis=(0, 1))


def normalise_saliency(T: np.ndarray, prunable: np.ndarray, mode: str = "max") -> np.ndarray:
    """Appendix "Combination with token-level importance": H_i is normalised to [0, H_max].
    Reading: T_hat = T / max_{j prunable} T_j (H_max = 1); unchanged when there is no prunable
    token or the maximum is not positive; mode "none" leaves T as is."""
    T = np.asarray(T, dtype=np.float64)
    if mode == "none":
        return T.copy()
    m = T[prunable].max() if prunable.any() else 0.0
    return T / m if m > 0 else T.copy()


# --------------------------------------------------------------------------------------
# Stages 2-3: step utility (Sec. 4.1, Eqs. 2-4) and retention priority (Eq. 5)
# --------------------------------------------------------------------------------------
def completion_score(valid, gain, red, lam: float) -> np.ndarray:
    """Eq. 2: r_k = valid_k + gain_k - lambda * red_k."""
    return np.asarray(valid, np.float64) + np.asarray(gain, np.float64) - lam * np.asarray(red, np.float64)


def reuse_update(c_prev, obs_sim, eta: float) -> np.ndarray:
    """Algorithm 1 Phase 1 (c_t <- 0 for the new step t = n_steps-1) and Phase 2 (Eq. 3:
    c_k <- c_k + min(1, eta * sim(Obs_t, Obs_k)) for 1 <= k < t).  obs_sim=None: no update."""
    c = np.asarray(c_prev, dtype=np.float64).copy()
    t = c.shape[0] - 1
    if t < 0:
        return c
    c[t] = 0.0
    if obs_sim is not None:
        sim = np.asarray(obs_sim, dtype=np.float64)
        for k in range(t):
            c[k] = c[k] + min(1.0, eta * sim[k])
    return c


def cue_similarity(a, b) -> float:
    """sim(a, b) of Sec. 4.1, "overlap-based textual similarity" over evidence cues (at most 64 per field,
    Table H).  Reading: the overlap of the two cue sets relative to their union, |A n B| / |A u B|, and 0
    when both are empty."""
    A, B = set(int(x) for x in a), set(int(x) for x in b)
    union = len(A | B)
    return len(A & B) / union if union else 0.0


def step_signals(th, act, obs, k0=None):
    """Sec. 4.1 field signals from per-step cue sets th[k], act[k], obs[k] (k = 0 .. t, t the newest step):
      gain_k = 1 - max_{u<k} sim(Th_k || Obs_k, Th_u || Obs_u)  (gain = 1 for the first step)
      red_k  = max_{u<k} sim(Act_k, Act_u)                       (red = 0 for the first step)
    for k >= k0 (default: the newest step only), and Eq. 3's obs_sim[k] = sim(Obs_t, Obs_k) for k < t
    (obs_sim[t] = 0).  The concatenation of two fields is the union of their cues (reading)."""
    n = len(obs)
    t = n - 1
    k0 = t if k0 is None else k0
    gain = np.full(n, np.nan)
    red = np.full(n, np.nan)
    for k in range(k0, n):
        cur = set(th[k]) | set(obs[k])
        gain[k] = 1.0 - max([cue_similarity(cur, set(th[u]) | set(obs[u])) for u in range(k)], default=0.0)
        red[k] = max([cue_similarity(act[k], act[u]) for u in range(k)], default=0.0)
    obs_sim = np.zeros(n)
    for k in range(t):
        obs_sim[k] = cue_similarity(obs[t], obs[k])
    return gain, red, obs_sim


def clip(z, a, b):
    """clip(z, a, b) truncates z to [a, b] (Sec. 4.1)."""
    return np.minimum(np.maximum(z, a), b)


def step_utility(r, c, p: Params) -> np.ndarray:
    """Eq. 4: S_k = clip(w_r * clip(r_k, r_min, r_max) + w_c * log(1 + c_k), 0, S_max), natural log."""
    r = np.asarray(r, np.float64)
    c = np.asarray(c, np.float64)
    return clip(p.w_r * clip(r, p.r_min, p.r_max) + p.w_c * np.log1p(c), 0.0, p.s_max)


def priority(T_hat, S, step_id, prunable, p: Params) -> np.ndarray:
    """Eq. 5: P_i = alpha * T_i + beta * S_{s(i)} for token i of step s(i); protected tokens are
    not ranked (reported as -inf)."""
    T_hat = np.asarray(T_hat, np.float64)
    P = np.full(T_hat.shape, -np.inf)
    idx = np.nonzero(prunable)[0]
    P[idx] = p.alpha * T_hat[idx] + p.beta * np.asarray(S, np.float64)[step_id[idx]]
    return P


# --------------------------------------------------------------------------------------
# Stage 4: budget and global top-B (Eq. 1; Sec. 4.2 "globally ranks tokens by P_i and
# retains the top B_t"; Algorithm 1 Phase 3)
# --------------------------------------------------------------------------------------
def budget_tokens(N: int, mode: str, num: int = 1, den: int = 1, count: int = 0) -> int:
    """Eq. 1: B_t = max(1, floor(rho * N_t)) with rho = num/den (exact rational), and |K| <= B_t,
    read as |K| = min(B_t, N_t) (0 when N_t = 0).  A fixed count budget gives B directly."""
    if N <= 0:
        return 0
    if mode == "ratio":
        B = max(1, (num * N) // den)
    elif mode == "count":
        B = int(count)
    else:
        raise ValueError(mode)
    return min(B, N)


def select_top(P: np.ndarray, prunable: np.ndarray, B: int) -> np.ndarray:
    """Indices of the B prunable tokens with the largest P, ties broken by the smaller index
    (reading: the older token wins), returned in ascending index order."""
    idx = np.nonzero(prunable)[0]
    order = np.lexsort((idx, -P[idx]))        # primary key -P (desc P), secondary key index (asc)
    return np.sort(idx[order[:B]])


def kept_indices(prot: np.ndarray, chosen: np.ndarray) -> np.ndarray:
    """Eq. 1: C_hat = C_prot || C_traj[K]; the retained slots in ascending original order."""
    keep = np.asarray(prot, dtype=bool).copy()
    keep[chosen] = True
    return np.nonzero(keep)[0].astype(np.int64)


# --------------------------------------------------------------------------------------
# Stage 5: compaction (Eq. 1: the compressed cache is the retained rows, densely packed)
# --------------------------------------------------------------------------------------
def compact_rows(X: np.ndarray, kept: np.ndarray) -> np.ndarray:
    """X: [H, T, d] (any dtype) -> [H, n_kept, d] with row r = X[:, kept[r], :]."""
    return np.asarray(X)[:, kept, :].copy()


def step_statistics(T_hat, step_id, prunable, chosen, n_steps: int) -> Dict[str, np.ndarray]:
    """Per-step accounting over prunable tokens (the evicted/retained-by-step view of Figs. 2 and 8):
    token count, sum and max of normalised saliency, and retained count.  Keyed by each token's own
    step id; protected tokens enter no figure; a step with no prunable token reports zeros."""
    T_hat = np.asarray(T_hat, np.float64)
    count = np.zeros(n_steps, np.int64)
    ssum = np.zeros(n_steps, np.float64)
    smax = np.zeros(n_steps, np.float64)
    kept = np.zeros(n_steps, np.int64)
    chosen_mask = np.zeros(T_hat.shape[0], bool)
    chosen_mask[chosen] = True
    for i in np.nonzero(prunable)[0]:
        k = int(step_id[i])
        count[k] += 1
        ssum[k] += T_hat[i]
        smax[k] = max(smax[k], T_hat[i])
        kept[k] += int(chosen_mask[i])
    return {"count": count, "sal_sum": ssum, "sal_max": smax, "kept": kept}


# --------------------------------------------------------------------------------------
# One pruning boundary, in Algorithm 1's order
# --------------------------------------------------------------------------------------
def stepkv_boundary(A_layers: Sequence[np.ndarray], step_id: np.ndarray, prot: np.ndarray,
                    valid, gain, red, obs_sim, reuse_prev, p: Params, budget_mode: str,
                    num: int = 1, den: int = 1, count: int = 0) -> Dict[str, np.ndarray]:
    """Algorithm 1 at the boundary after step t = n_steps-1, given per-layer saliency A.

    Phase 1: r_t (Eq. 2), c_t <- 0, S_t (Eq. 4).  Phase 2: for k < t update c_k (Eq. 3) and
    recompute S_k (Eq. 4).  Phase 3: B_t (Eq. 1), P_i (Eq. 5), top-B_t by P_i.
    """
    step_id = np.asarray(step_id)
    prot = np.asarray(prot).astype(bool)
    prunable = ~prot
    n_steps = len(valid)
    # Phase 1 + 2 (the r_k of earlier steps are recomputed from their stored signals)
    r = completion_score(valid, gain, red, p.lam)
    c = reuse_update(reuse_prev, obs_sim, p.eta)
    S = step_utility(r, c, p)
    # Phase 3
    T_raw = token_saliency(A_layers, p.pool, p.pool_mode)
    T_hat = normalise_saliency(T_raw, prunable, p.sal_norm)
    N = int(prunable.sum())
    B = budget_tokens(N, budget_mode, num, den, count)
    P = priority(T_hat, S, step_id, prunable, p)
    chosen = select_top(P, prunable, B)
    kept = kept_indices(prot, chosen)
    stats = step_statistics(T_hat, step_id, prunable, chosen, n_steps)
    return {"r": r, "reuse": c, "S": S, "T": T_raw, "T_hat": T_hat, "N": N, "B": B, "P": P,
            "chosen": chosen, "kept": kept, **{"step_" + k: v for k, v in stats.items()}}


def compress(K_sal: Sequence[np.ndarray], Q_sal: Sequence[np.ndarray], step_id, prot, valid, gain, red,
             obs_sim, reuse_prev, p: Params, budget_mode: str, num: int = 1, den: int = 1,
             count: int = 0) -> Dict[str, np.ndarray]:
    """Score -> select for one trajectory: saliency from the last layers' window queries, then
    Algorithm 1.  Compaction of any layer is ``compact_rows(X, out['kept'])``."""
    A = [window_attention_saliency(k, q) for k, q in zip(K_sal, Q_sal)]
    out = stepkv_boundary(A, step_id, prot, valid, gain, red, obs_sim, reuse_prev, p, budget_mode,
                          num, den, count)
    out["A"] = np.stack(A)
    return out


def decode_attention(q: np.ndarray, K: np.ndarray, V: np.ndarray) -> np.ndarray:
    """Single-token attention over a (compacted) cache, GQA: q [Hq, d], K/V [Hkv, n, d] bf16 bits ->
    out [Hq, d] float64 = softmax(q.K^T / sqrt(d)) V per q head, with q head g reading KV head g // G."""
    qf = bf16_to_f64(q)
    Kf = bf16_to_f64(K)
    Vf = bf16_to_f64(V)
    Hq, d = qf.shape
    Hkv = Kf.shape[0]
    G = Hq // Hkv
    out = np.zeros((Hq, d))
    for g in range(Hq):
        h = g // G
        s = Kf[h] @ qf[g] / math.sqrt(d)
        s = s - s.max()
        e = np.exp(s)
        out[g] = (e / e.sum()) @ Vf[h]
    return out


def decode_attention_mass(q: np.ndarray, K: np.ndarray) -> np.ndarray:
    """Accumulated-attention token saliency of one decode read (Sec. 4.2: T_i "can be supplied by existing
    token-level KV importance estimators"; H2O scores a token by the attention mass it receives).
    q [Hq, d], K [Hkv, n, d] bf16 bits -> A [Hkv, n] float64 with
        A[h, j] = (1/G) * sum_{g in group(h)} softmax_j(q_g . K[h, j] / sqrt(d)),
    the softmax weight key j receives from the group's query heads (mean over the GQA group, as for the
    window saliency).  Summed over the decode reads between two boundaries it is the H2O score."""
    qf = bf16_to_f64(q)
    Kf = bf16_to_f64(K)
    Hq, d = qf.shape
    Hkv, n, _ = Kf.shape
    G = Hq // Hkv
    A = np.zeros((Hkv, n))
    for g in range(Hq):
        h = g // G
        s = Kf[h] @ qf[g] / math.sqrt(d)
        s = s - s.max()
        e = np.exp(s)
        A[h] += e / e.sum()
    return A / G
