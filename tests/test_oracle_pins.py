"""Pins for the CPU oracle: each check ties an oracle function to something other than itself
(hand-computed tables, closed forms, textbook/library special cases, brute force, invariants).

Every check is written as ``check_*(O)`` taking an oracle-like namespace, so the planted-mistake
tests at the bottom can run the same check against a deliberately broken copy of the oracle and
confirm that the check fails.  CPU only.
"""
import itertools
import math
import os
import types

import numpy as np
import pytest
from scipy.special import expit, softmax

from oracle import stepkv_oracle as REAL
from paper_2609_22158_gb300 import workload as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _load_table(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


def _bits(x):
    return wl.f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


# ------------------------------------------------------------------ Eqs. 2-4 (hand tables)
def check_step_utility_table(O):
    p = O.Params()
    for case, valid, gain, red, logc, er, es in _load_table("eq2_4_table_h.txt"):
        valid, gain, red, logc, er, es = map(float, (valid, gain, red, logc, er, es))
        r = O.completion_score([valid], [gain], [red], p.lam)[0]
        assert abs(r - er) < 1e-12, (case, r, er)
        S = O.step_utility([r], [math.expm1(logc)], p)[0]
        assert abs(S - es) < 1e-12, (case, S, es)


def check_s_max_clip(O):
    p = O.Params(w_c=10.0)
    S = O.step_utility([2.0], [math.expm1(2.0)], p)[0]      # 0.85*2 + 10*2 = 21.7 -> 8
    assert S == 8.0


def check_reuse_table(O):
    rows = _load_table("eq3_reuse.txt")
    c_prev = [float(r[1]) for r in rows]
    sim = [float(r[2]) for r in rows]
    exp = [float(r[3]) for r in rows]
    c = O.reuse_update(c_prev, sim, O.Params().eta)
    assert np.allclose(c, exp, rtol=0, atol=1e-12), (c, exp)
    # no similarity vector: only the Phase-1 reset of the new step
    c2 = O.reuse_update(c_prev, None, 1.5)
    assert np.allclose(c2, [0.5, 0.0, 2.0, 0.0])


def test_step_utility_table():
    check_step_utility_table(REAL)


def test_s_max_clip():
    check_s_max_clip(REAL)


def test_reuse_table():
    check_reuse_table(REAL)


def test_step_utility_invariants():
    # Eq. 4 range [0, S_max] and c_k >= 0 with increments <= 1 (appendix "Step Score")
    rng = np.random.default_rng(5)
    p = REAL.Params()
    for _ in range(20):
        n = 50
        valid = (rng.random(n) > 0.3).astype(float)
        gain, red, sim = rng.random(n), rng.random(n) * 3, rng.random(n) * 2
        c0 = rng.random(n) * 5
        c = REAL.reuse_update(c0, sim, p.eta)
        assert (c >= 0).all()
        assert (c[:-1] - c0[:-1] <= 1 + 1e-15).all() and (c[:-1] >= c0[:-1]).all()
        S = REAL.step_utility(REAL.completion_score(valid, gain, red, p.lam), c, p)
        assert (S >= 0).all() and (S <= p.s_max).all()


# ------------------------------------------------------------------ saliency closed forms
def _rand_qk(rng, Hkv, G, T, W, d):
    K = _bits(rng.standard_normal((Hkv, T, d)))
    Q = _bits(rng.standard_normal((Hkv * G, W, d)))
    return K, Q


def check_zero_keys_closed_form(O):
    """K == 0: every visible logit is 0, so query w (slot p_w = T-W+w) spreads 1/(p_w+1) uniformly
    over keys j <= p_w; A[h, j] = sum_w [j <= p_w] / (p_w + 1), for every head and any queries."""
    rng = np.random.default_rng(1)
    for (Hkv, G, T, W, d) in [(2, 3, 50, 7, 16), (1, 1, 9, 9, 8), (3, 2, 40, 1, 32)]:
        K = np.zeros((Hkv, T, d), np.uint16)
        Q = _bits(rng.standard_normal((Hkv * G, W, d)))
        A = O.window_attention_saliency(K, Q)
        exp = np.zeros(T)
        for w in range(W):
            pw = T - W + w
            exp[:pw + 1] += 1.0 / (pw + 1)
        for h in range(Hkv):
            assert np.allclose(A[h], exp, rtol=1e-12, atol=1e-15), (Hkv, G, T, W)


def check_mass_conservation(O):
    """Each window query's softmax sums to 1, so sum_j A[h, j] = W (mean over the group)."""
    rng = np.random.default_rng(2)
    K, Q = _rand_qk(rng, 2, 4, 300, 13, 32)
    A = O.window_attention_saliency(K, Q)
    assert np.allclose(A.sum(axis=1), 13.0, rtol=1e-12)


def check_single_query_softmax(O):
    """W = 1, G = 1: the one query sits at slot T-1 and sees every key, so A[h] is the textbook
    softmax of q.K^T / sqrt(d) (scipy)."""
    rng = np.random.default_rng(3)
    for d in (16, 64, 128):
        K, Q = _rand_qk(rng, 3, 1, 257, 1, d)
        A = O.window_attention_saliency(K, Q)
        Kf, Qf = REAL.bf16_to_f64(K), REAL.bf16_to_f64(Q)
        for h in range(3):
            ref = softmax(Kf[h] @ Qf[h, 0] / math.sqrt(d))
            assert np.allclose(A[h], ref, rtol=1e-12, atol=1e-300)


def check_two_key_analytic(O):
    """T=2, W=1: q=(1,0,0,0), k0=(2,0,0,0), k1=0, d=4: logits 2/sqrt(4)=1 and 0, so
    A = (sigmoid(1), sigmoid(-1))."""
    K = _bits([[[2, 0, 0, 0], [0, 0, 0, 0]]])
    Q = _bits([[[1, 0, 0, 0]]])
    A = O.window_attention_saliency(K, Q)
    assert np.allclose(A[0], [expit(1.0), expit(-1.0)], rtol=1e-14)


def check_gqa_grouping(O):
    """q heads h*G..h*G+G-1 read KV head h.  KV head 1 is all zeros, so A[1] must be the uniform
    closed form whatever its group's queries are; A[0] must be the mean over q heads 0..G-1 of
    their own softmaxes against K[0] (last query sees everything; W=1)."""
    rng = np.random.default_rng(4)
    G, T, d = 2, 64, 16
    K = np.zeros((2, T, d), np.uint16)
    K[0] = _bits(rng.standard_normal((T, d)) * 2)
    Q = _bits(rng.standard_normal((4, 1, d)) * 2)
    A = O.window_attention_saliency(K, Q)
    Kf, Qf = REAL.bf16_to_f64(K), REAL.bf16_to_f64(Q)
    ref0 = np.mean([softmax(Kf[0] @ Qf[g, 0] / math.sqrt(d)) for g in (0, 1)], axis=0)
    assert np.allclose(A[0], ref0, rtol=1e-12)
    assert np.allclose(A[1], np.full(T, 1.0 / T), rtol=1e-12)


def check_causal_last_key(O):
    """Key at slot T-1 is visible only to the last window query: A[h, T-1] equals the mean over
    the group of that query's softmax weight on it."""
    rng = np.random.default_rng(6)
    G, T, W, d = 3, 40, 5, 16
    K, Q = _rand_qk(rng, 1, G, T, W, d)
    A = O.window_attention_saliency(K, Q)
    Kf, Qf = REAL.bf16_to_f64(K), REAL.bf16_to_f64(Q)
    ref = np.mean([softmax(Kf[0] @ Qf[g, W - 1] / math.sqrt(d))[T - 1] for g in range(G)])
    assert abs(A[0, T - 1] - ref) <= 1e-12 * ref


@pytest.mark.parametrize("chk", [check_zero_keys_closed_form, check_mass_conservation, check_single_query_softmax,
                                 check_two_key_analytic, check_gqa_grouping, check_causal_last_key])
def test_saliency_pins(chk):
    chk(REAL)


def test_token_saliency_mean_and_normalisation():
    A = [np.array([[1.0, 2.0, 3.0, 9.0]]), np.array([[3.0, 2.0, 1.0, 9.0]])]
    T = REAL.token_saliency(A)
    assert np.allclose(T, [2.0, 2.0, 2.0, 9.0])
    prunable = np.array([True, True, True, False])       # protected token holds the largest value
    That = REAL.normalise_saliency(T, prunable, "max")
    assert np.allclose(That, [1.0, 1.0, 1.0, 4.5])      # max over prunable tokens only
    assert np.allclose(REAL.normalise_saliency(T, prunable, "none"), T)
    assert np.allclose(REAL.normalise_saliency(T, np.zeros(4, bool), "max"), T)


# ------------------------------------------------------------------ budget (Eq. 1)
def check_budget(O):
    assert O.budget_tokens(2000, "ratio", 1, 4) == 500
    assert O.budget_tokens(32688, "ratio", 1, 10) == 3268
    assert O.budget_tokens(3, "ratio", 1, 10) == 1          # max(1, floor(0.3))
    assert O.budget_tokens(0, "ratio", 1, 2) == 0            # nothing prunable: K is empty
    assert O.budget_tokens(100, "count", count=4096) == 100  # |K| <= N
    assert O.budget_tokens(10, "ratio", 7, 7) == 10
    assert O.budget_tokens(9, "ratio", 1, 3) == 3


def test_budget():
    check_budget(REAL)


# ------------------------------------------------------------------ global top-B selection
def _dominance_ok(P, prunable, K):
    Ks = set(K.tolist())
    for i in Ks:
        for j in np.nonzero(prunable)[0]:
            if j in Ks:
                continue
            if not (P[i] > P[j] or (P[i] == P[j] and i < j)):
                return False
    return True


def check_select_bruteforce(O):
    """Enumerate every subset of size B of the prunable tokens; exactly one keeps each retained
    token ahead of each evicted one under (P desc, index asc), and it is the oracle's set."""
    rng = np.random.default_rng(7)
    for trial in range(25):
        N = int(rng.integers(1, 10))
        P = rng.choice([0.0, 0.25, 0.5, 0.75, 1.0], size=N)   # many ties
        prunable = rng.random(N) > 0.25
        idx = np.nonzero(prunable)[0]
        for B in range(0, len(idx) + 1):
            valid = [np.array(c, dtype=np.int64) for c in itertools.combinations(idx, B)
                     if _dominance_ok(P, prunable, np.array(c, dtype=np.int64))]
            assert len(valid) == 1
            got = O.select_top(P, prunable, B)
            assert np.array_equal(got, valid[0]), (P, prunable, B, got, valid[0])


def check_select_rank_count(O):
    """O(N^2) rank counting: token i is kept iff fewer than B prunable tokens beat it
    (larger P, or equal P and smaller index)."""
    rng = np.random.default_rng(8)
    for N in (50, 400, 1500):
        P = np.round(rng.random(N) * 40) / 40                   # ties
        prunable = rng.random(N) > 0.1
        idx = np.nonzero(prunable)[0]
        Pi = P[idx]
        beats = (Pi[None, :] > Pi[:, None]) | ((Pi[None, :] == Pi[:, None]) & (idx[None, :] < idx[:, None]))
        rank = beats.sum(axis=1)
        for B in (0, 1, len(idx) // 3, len(idx)):
            exp = np.sort(idx[rank < B])
            assert np.array_equal(O.select_top(P, prunable, B), exp)


def test_select_pins():
    check_select_bruteforce(REAL)
    check_select_rank_count(REAL)


def test_ablation_special_cases():
    """Table 3 ablations: alpha=0 ranks by step utility alone (ties inside a step fall to the older
    tokens); beta=0 is plain saliency top-k."""
    rng = np.random.default_rng(9)
    T, n_steps = 300, 6
    step_id = np.repeat(np.arange(n_steps), T // n_steps).astype(np.int32)
    prunable = np.ones(T, bool)
    prunable[:5] = False
    T_hat = rng.random(T)
    S = np.array([0.3, 1.5, 0.1, 1.1, 0.9, 0.2])
    B = 77
    p0 = REAL.Params(alpha=0.0, beta=1.0)
    got = REAL.select_top(REAL.priority(T_hat, S, step_id, prunable, p0), prunable, B)
    # expected: walk steps by descending S, taking tokens in index order
    exp = []
    for k in np.argsort(-S, kind="stable"):
        for i in np.nonzero((step_id == k) & prunable)[0]:
            if len(exp) < B:
                exp.append(i)
    assert np.array_equal(got, np.sort(exp))
    p1 = REAL.Params(alpha=1.0, beta=0.0)
    got = REAL.select_top(REAL.priority(T_hat, S, step_id, prunable, p1), prunable, B)
    idx = np.nonzero(prunable)[0]
    assert np.array_equal(got, np.sort(idx[np.argsort(-T_hat[idx], kind="stable")[:B]]))


def test_priority_range_and_sharing():
    """Eq. 5 / appendix score range: P in [0, alpha*1 + beta*S_max] with T_hat in [0,1];
    tokens of one step share S_k, so P differences inside a step are alpha*(T_i - T_j)."""
    rng = np.random.default_rng(10)
    p = REAL.Params()
    T = 200
    step_id = np.repeat(np.arange(4), 50).astype(np.int32)
    prunable = np.ones(T, bool)
    T_hat = rng.random(T)
    S = np.array([0.0, 8.0, 3.0, 1.0])
    P = REAL.priority(T_hat, S, step_id, prunable, p)
    assert (P >= 0).all() and (P <= p.alpha + p.beta * p.s_max).all()
    i, j = 60, 70
    assert abs((P[i] - P[j]) - p.alpha * (T_hat[i] - T_hat[j])) < 1e-12


# ------------------------------------------------------------------ decode attention (S6)
def check_decode_single_key(O):
    # one cached key: the softmax weight is 1 and the output is that key's value row, exactly
    rng = np.random.default_rng(7)
    q = _bits(rng.standard_normal((4, 16)))
    K = _bits(rng.standard_normal((2, 1, 16)))
    V = _bits(rng.standard_normal((2, 1, 16)))
    out = O.decode_attention(q, K, V)
    Vf = O.bf16_to_f64(V)
    for g in range(4):
        assert np.array_equal(out[g], Vf[g // 2, 0])


def check_decode_identical_keys(O):
    # equal keys: uniform weights, the output is the mean of the value rows
    rng = np.random.default_rng(8)
    k = rng.standard_normal(32)
    K = _bits(np.tile(k, (1, 9, 1)))
    V = _bits(rng.standard_normal((1, 9, 32)))
    q = _bits(rng.standard_normal((3, 32)))
    out = O.decode_attention(q, K, V)
    mean = O.bf16_to_f64(V)[0].mean(axis=0)
    assert np.allclose(out, np.tile(mean, (3, 1)), rtol=0, atol=1e-12)


def check_decode_two_key_analytic(O):
    # two keys: the first weight is the logistic function of the scaled logit difference
    d = 16
    q = np.zeros((1, d), np.float32)
    q[0, 0] = 2.0
    K = np.zeros((1, 2, d), np.float32)
    K[0, 0, 0] = 1.5
    K[0, 1, 0] = -0.5
    V = np.zeros((1, 2, d), np.float32)
    V[0, 0, 3] = 1.0
    V[0, 1, 5] = 1.0
    out = O.decode_attention(_bits(q), _bits(K), _bits(V))
    w0 = expit((2.0 * 1.5 - 2.0 * -0.5) / math.sqrt(d))
    assert abs(out[0, 3] - w0) < 1e-12 and abs(out[0, 5] - (1 - w0)) < 1e-12
    assert abs(out[0].sum() - 1.0) < 1e-12


def check_decode_gqa(O):
    # query head g reads KV head g // G: value rows are constant per KV head
    d, n = 8, 5
    rng = np.random.default_rng(9)
    q = _bits(rng.standard_normal((6, d)))
    K = _bits(rng.standard_normal((3, n, d)))
    V = np.stack([np.full((n, d), 1.0 + h, np.float32) for h in range(3)])
    out = O.decode_attention(q, K, _bits(V))
    for g in range(6):
        assert np.allclose(out[g], 1.0 + g // 2, rtol=0, atol=1e-12)


def check_decode_bruteforce(O):
    # element-by-element restatement with math.exp on a tiny case
    rng = np.random.default_rng(10)
    Hq, Hkv, n, d = 4, 2, 6, 4
    q = _bits(rng.standard_normal((Hq, d)))
    K = _bits(rng.standard_normal((Hkv, n, d)))
    V = _bits(rng.standard_normal((Hkv, n, d)))
    qf, Kf, Vf = (O.bf16_to_f64(x) for x in (q, K, V))
    out = O.decode_attention(q, K, V)
    for g in range(Hq):
        h = g * Hkv // Hq
        logits = [sum(qf[g][t] * Kf[h][j][t] for t in range(d)) / math.sqrt(d) for j in range(n)]
        mx = max(logits)
        w = [math.exp(x - mx) for x in logits]
        z = sum(w)
        for t in range(d):
            ref = sum(w[j] / z * Vf[h][j][t] for j in range(n))
            assert abs(out[g][t] - ref) < 1e-12


def test_decode_single_key():
    check_decode_single_key(REAL)


def test_decode_identical_keys():
    check_decode_identical_keys(REAL)


def test_decode_two_key_analytic():
    check_decode_two_key_analytic(REAL)


def test_decode_gqa():
    check_decode_gqa(REAL)


def test_decode_bruteforce():
    check_decode_bruteforce(REAL)


# ------------------------------------------------------------------ accumulated decode attention (H2O-style)
def check_mass_single_query_softmax(O):
    """One KV head, one query head: the mass is the textbook softmax of the scaled logits (scipy)."""
    rng = np.random.default_rng(31)
    q, K = _bits(rng.standard_normal((1, 16))), _bits(rng.standard_normal((1, 37, 16)))
    A = O.decode_attention_mass(q, K)
    ref = softmax(REAL.bf16_to_f64(K)[0] @ REAL.bf16_to_f64(q)[0] / 4.0)
    assert np.allclose(A[0], ref, rtol=1e-12, atol=0)


def check_mass_sums(O):
    """Every KV head receives a total of exactly one per read (each query head's softmax sums to one, and
    the group's heads are averaged); summed over reads, the masses total the number of reads."""
    rng = np.random.default_rng(32)
    Hkv, G, n, d = 3, 4, 50, 32
    tot = np.zeros((Hkv, n))
    for r in range(5):
        A = O.decode_attention_mass(_bits(rng.standard_normal((Hkv * G, d))), _bits(rng.standard_normal((Hkv, n, d))))
        assert np.allclose(A.sum(axis=1), 1.0, rtol=0, atol=1e-12)
        assert (A >= 0).all()
        tot += A
    assert np.allclose(tot.sum(axis=1), 5.0, rtol=0, atol=1e-11)


def check_mass_two_key_analytic(O):
    """Two keys: the first key's weight is the logistic function of the scaled logit difference."""
    q = _bits(np.full((1, 16), 0.5))
    K = _bits(np.stack([np.full(16, 1.0), np.full(16, -0.5)])[None])
    A = O.decode_attention_mass(q, K)
    s0, s1 = 16 * 0.5 * 1.0 / 4.0, 16 * 0.5 * -0.5 / 4.0
    assert abs(A[0, 0] - expit(s0 - s1)) < 1e-14 and abs(A[0, 1] - expit(s1 - s0)) < 1e-14


def check_mass_gqa(O):
    """Query head g reads KV head g // G: a group whose heads all match key 0 puts its mass there."""
    d, n = 16, 4
    K = np.zeros((2, n, d), np.float32)
    K[0, 0, 0] = K[0, 1, 1] = 8.0   # KV head 0: key 0 along e0, key 1 along e1
    K[1, 2, 0] = K[1, 3, 1] = 8.0   # KV head 1: key 2 along e0, key 3 along e1
    q = np.zeros((4, d), np.float32)  # G = 2: heads 0, 1 -> KV head 0; heads 2, 3 -> KV head 1
    q[0, 0] = q[1, 0] = 8.0           # group of KV head 0 looks along e0
    q[2, 1] = q[3, 1] = 8.0           # group of KV head 1 looks along e1
    A = O.decode_attention_mass(_bits(q), _bits(K))
    assert A[0, 0] > 0.99 and A[1, 3] > 0.99


def check_mass_bruteforce(O):
    """Plain loops over heads and keys, exponentials and sums written out, on a tiny case."""
    rng = np.random.default_rng(33)
    Hkv, G, n, d = 2, 2, 5, 4
    q, K = _bits(rng.standard_normal((Hkv * G, d))), _bits(rng.standard_normal((Hkv, n, d)))
    qf, Kf = REAL.bf16_to_f64(q), REAL.bf16_to_f64(K)
    ref = np.zeros((Hkv, n))
    for g in range(Hkv * G):
        h = g // G
        logits = [sum(qf[g, e] * Kf[h, j, e] for e in range(d)) / math.sqrt(d) for j in range(n)]
        ex = [math.exp(x) for x in logits]
        tot = sum(ex)
        for j in range(n):
            ref[h, j] += ex[j] / tot / G
    assert np.allclose(O.decode_attention_mass(q, K), ref, rtol=1e-12, atol=0)


@pytest.mark.parametrize("chk", [check_mass_single_query_softmax, check_mass_sums, check_mass_two_key_analytic,
                                 check_mass_gqa, check_mass_bruteforce])
def test_decode_mass_pins(chk):
    chk(REAL)


# ------------------------------------------------------------------ step signals from evidence cues (Sec. 4.1)
def _signal_table():
    rows = _load_table("step_signals.txt")
    parse = lambda x: [] if x == "-" else [int(v) for v in x.split(",")]
    steps = [r[1:] for r in rows if r[0] == "step"]
    sig = np.array([[float(v) for v in r[2:]] for r in rows if r[0] == "sig"])
    return [parse(r[1]) for r in steps], [parse(r[2]) for r in steps], [parse(r[3]) for r in steps], sig


def check_step_signals_table(O):
    th, act, obs, sig = _signal_table()
    gain, red, obs_sim = O.step_signals(th, act, obs, k0=0)
    assert np.allclose(gain, sig[:, 0], rtol=0, atol=1e-15), gain
    assert np.allclose(red, sig[:, 1], rtol=0, atol=1e-15), red
    assert np.allclose(obs_sim, sig[:, 2], rtol=0, atol=1e-15), obs_sim


def check_cue_similarity_cases(O):
    """Identical non-empty sets give 1, disjoint or empty sets 0, the value is symmetric, and it equals
    a count written out with loops on random small sets."""
    assert O.cue_similarity([3, 5, 9], [3, 5, 9]) == 1.0
    assert O.cue_similarity([3, 5], [4, 6]) == 0.0
    assert O.cue_similarity([], []) == 0.0 and O.cue_similarity([1], []) == 0.0
    rng = np.random.default_rng(9)
    for _ in range(50):
        a = sorted(set(rng.integers(0, 30, rng.integers(0, 12)).tolist()))
        b = sorted(set(rng.integers(0, 30, rng.integers(0, 12)).tolist()))
        inter = sum(1 for x in a if x in b)
        union = len(a) + sum(1 for x in b if x not in a)
        ref = inter / union if union else 0.0
        assert O.cue_similarity(a, b) == ref and O.cue_similarity(b, a) == ref


def test_step_signals_table():
    check_step_signals_table(REAL)


def test_cue_similarity_cases():
    check_cue_similarity_cases(REAL)


def test_step_signals_ranges():
    rng = np.random.default_rng(10)
    draw = lambda: sorted(set(rng.integers(0, 200, rng.integers(0, 64)).tolist()))
    th, act, obs = [draw() for _ in range(30)], [draw() for _ in range(30)], [draw() for _ in range(30)]
    gain, red, obs_sim = REAL.step_signals(th, act, obs, k0=0)
    assert gain[0] == 1.0 and red[0] == 0.0 and obs_sim[-1] == 0.0
    assert ((gain >= 0) & (gain <= 1)).all() and ((red >= 0) & (red <= 1)).all()
    assert ((obs_sim >= 0) & (obs_sim <= 1)).all()


# ------------------------------------------------------------------ end-to-end invariants
def test_boundary_invariants_tiny():
    tr = wl.tiny(0)
    s = tr.shape
    p = REAL.Params()
    Ks = [tr.keys(l) for l in tr.sal_layer_ids()]
    Qs = [tr.queries(l) for l in tr.sal_layer_ids()]
    out = REAL.compress(Ks, Qs, tr.step_id, tr.prot, tr.valid, tr.gain, tr.red, tr.obs_sim, tr.reuse, p,
                        tr.budget.mode, tr.budget.num, tr.budget.den, tr.budget.count)
    prot = tr.prot.astype(bool)
    N = int((~prot).sum())
    assert out["N"] == N == 2048 - 16 - 32
    assert out["B"] == N // 4 == 500
    kept = out["kept"]
    assert len(kept) == int(prot.sum()) + out["B"]
    assert np.all(np.diff(kept) > 0)
    assert set(np.nonzero(prot)[0]).issubset(set(kept.tolist()))
    assert out["step_kept"].sum() == out["B"] and out["step_count"].sum() == N
    assert (out["S"] >= 0).all() and (out["S"] <= p.s_max).all()
    assert out["reuse"][-1] == 0.0
    assert abs(out["T_hat"][~prot].max() - 1.0) < 1e-15
    assert np.allclose(out["A"].sum(axis=2), s.W)
    V = tr.values(0)
    C = REAL.compact_rows(V, kept)
    for r in range(0, len(kept), 37):
        assert np.array_equal(C[:, r, :], V[:, kept[r], :])


# ------------------------------------------------------------------ per-step accounting (hand table)
def _step_table():
    rows = _load_table("step_statistics.txt")
    tok = [r[1:] for r in rows if r[0] == "tok"]
    step = [r[1:] for r in rows if r[0] == "step"]
    step_id = np.array([int(r[1]) for r in tok], np.int32)
    prot = np.array([int(r[2]) for r in tok], np.uint8)
    T_raw = np.array([float(r[3]) for r in tok])
    T_hat = np.array([float(r[4]) for r in tok])
    exp = {"count": np.array([int(r[1]) for r in step]), "sal_sum": np.array([float(r[2]) for r in step]),
           "sal_max": np.array([float(r[3]) for r in step]), "kept": np.array([int(r[4]) for r in step])}
    return step_id, prot, T_raw, T_hat, exp


def _assert_step_stats(st, exp, prefix=""):
    assert np.array_equal(st[prefix + "count"], exp["count"]), (st[prefix + "count"], exp["count"])
    assert np.allclose(st[prefix + "sal_sum"], exp["sal_sum"], rtol=0, atol=1e-12), st[prefix + "sal_sum"]
    assert np.allclose(st[prefix + "sal_max"], exp["sal_max"], rtol=0, atol=1e-12), st[prefix + "sal_max"]
    assert np.array_equal(st[prefix + "kept"], exp["kept"]), (st[prefix + "kept"], exp["kept"])


def check_step_statistics_table(O):
    """step_statistics on the table's T_hat and retained set {4, 5, 9}."""
    step_id, prot, _, T_hat, exp = _step_table()
    st = O.step_statistics(T_hat, step_id, ~prot.astype(bool), np.array([4, 5, 9]), len(exp["count"]))
    _assert_step_stats(st, exp)


def check_boundary_step_statistics(O):
    """The whole boundary from raw saliency: normalisation over prunable tokens, alpha = 1, beta = 0,
    count budget 3 -- the per-step figures must be those of the table (computed on T_hat)."""
    step_id, prot, T_raw, T_hat, exp = _step_table()
    n = len(exp["count"])
    p = O.Params(alpha=1.0, beta=0.0)
    z = np.zeros(n)
    out = O.stepkv_boundary([T_raw[None, :]], step_id, prot, z + 1.0, z, z, None, z, p, "count", count=3)
    assert np.allclose(out["T_hat"], T_hat, rtol=0, atol=1e-15)
    assert out["N"] == 7 and out["B"] == 3 and list(out["chosen"]) == [4, 5, 9]
    _assert_step_stats(out, exp, prefix="step_")


def test_step_statistics_table():
    check_step_statistics_table(REAL)


def test_boundary_step_statistics():
    check_boundary_step_statistics(REAL)


# ------------------------------------------------------------------ prefill row log-sum-exp
def check_lse_zero_keys(O):
    """All logits 0: each row's log-sum-exp is log(number of visible keys) = log(T - W + w + 1)."""
    Hkv, G, T, W, d = 2, 2, 40, 6, 16
    K = _bits(np.zeros((Hkv, T, d)))
    Q = _bits(np.random.default_rng(1).standard_normal((Hkv * G, W, d)))
    lse = O.window_row_lse(K, Q)
    np.testing.assert_allclose(lse, np.log(T - W + np.arange(W) + 1.0)[None, :].repeat(Hkv * G, 0), rtol=1e-12)


def check_lse_logsumexp(O):
    """Brute force: scipy's logsumexp over each row's visible scaled dot products, key by key."""
    from scipy.special import logsumexp
    rng = np.random.default_rng(2)
    Hkv, G, T, W, d = 2, 3, 30, 4, 8
    K, Q = _rand_qk(rng, Hkv, G, T, W, d)
    Kf, Qf = wl.bf16_bits_to_f32(K).astype(np.float64), wl.bf16_bits_to_f32(Q).astype(np.float64)
    lse = O.window_row_lse(K, Q)
    for g in range(Hkv * G):
        for w in range(W):
            logits = [float(Qf[g, w] @ Kf[g // G, j]) / math.sqrt(d) for j in range(T - W + w + 1)]
            assert abs(lse[g, w] - logsumexp(logits)) < 1e-10


def check_lse_rebuilds_saliency(O):
    """exp(s - lse) summed over a KV head's query rows and averaged over its group is the saliency."""
    rng = np.random.default_rng(3)
    Hkv, G, T, W, d = 2, 2, 25, 5, 8
    K, Q = _rand_qk(rng, Hkv, G, T, W, d)
    Kf, Qf = wl.bf16_bits_to_f32(K).astype(np.float64), wl.bf16_bits_to_f32(Q).astype(np.float64)
    lse = O.window_row_lse(K, Q)
    A = np.zeros((Hkv, T))
    for g in range(Hkv * G):
        for w in range(W):
            vis = T - W + w + 1
            s = Qf[g, w] @ Kf[g // G, :vis].T / math.sqrt(d)
            A[g // G, :vis] += np.exp(s - lse[g, w]) / G
    np.testing.assert_allclose(A, O.window_attention_saliency(K, Q), rtol=1e-10, atol=1e-14)


def test_prefill_lse_pins():
    for chk in (check_lse_zero_keys, check_lse_logsumexp, check_lse_rebuilds_saliency):
        chk(REAL)


# ------------------------------------------------------------------ SnapKV-style pooling (Sec. 4.2)
def check_pool_table(O):
    """The hand table of tests/golden/snapkv_pooling.txt."""
    a = np.array([0.1, 0.5, 0.2, 0.0, 0.9, 0.3])
    for row in _load_table("snapkv_pooling.txt"):
        k, mode, exp = int(row[0]), row[1], np.array([float(x) for x in row[2:]])
        np.testing.assert_allclose(O.pool_tokens(a, k, mode), exp, rtol=0, atol=1e-12)


def check_pool_max_library(O):
    """Max pooling with the window clipped at the ends equals scipy's maximum filter with edge
    replication (a replicated edge value lies inside the clipped window)."""
    from scipy.ndimage import maximum_filter1d
    rng = np.random.default_rng(5)
    for T, k in ((1, 3), (2, 5), (7, 3), (50, 7), (33, 9)):
        a = rng.random(T)
        np.testing.assert_array_equal(O.pool_tokens(a, k, "max"), maximum_filter1d(a, size=k, mode="nearest"))


def check_pool_avg_convolution(O):
    """Average pooling: a k-tap box convolution where the whole window fits, the mean of the in-range
    values at the ends."""
    rng = np.random.default_rng(6)
    T, k = 40, 7
    h = k // 2
    a = rng.random(T)
    out = O.pool_tokens(a, k, "avg")
    np.testing.assert_allclose(out[h:T - h], np.convolve(a, np.ones(k) / k, mode="valid"), rtol=1e-12)
    for i in list(range(h)) + list(range(T - h, T)):
        assert abs(out[i] - a[max(0, i - h):min(T, i + h + 1)].mean()) < 1e-12


def check_pool_before_mean(O):
    """Each (layer, KV head) row is pooled before the mean over rows: for a maximum the two orders
    differ."""
    rows = [np.array([[1.0, 0.0, 0.0], [0.0, 0.0, 1.0]])]  # one layer, two KV heads
    np.testing.assert_allclose(O.token_saliency(rows, 3, "max"), [0.5, 1.0, 0.5])
    np.testing.assert_allclose(O.token_saliency(rows, 1, "max"), [0.5, 0.0, 0.5])


def test_snapkv_pooling_pins():
    for chk in (check_pool_table, check_pool_max_library, check_pool_avg_convolution, check_pool_before_mean):
        chk(REAL)


def test_boundary_uses_pooling():
    rng = np.random.default_rng(7)
    T, n_steps = 60, 4
    A = [rng.random((2, T)) for _ in range(2)]
    step_id = np.repeat(np.arange(n_steps), T // n_steps).astype(np.int32)
    prot = np.zeros(T, dtype=np.uint8)
    sig = [rng.random(n_steps) for _ in range(4)]
    p = REAL.Params(pool=5, pool_mode="avg")
    out = REAL.stepkv_boundary(A, step_id, prot, sig[0] > 0.5, sig[1], sig[2], sig[3], np.zeros(n_steps), p,
                               "ratio", 1, 4)
    np.testing.assert_allclose(out["T"], REAL.token_saliency(A, 5, "avg"))
    assert not np.allclose(out["T"], REAL.token_saliency(A))


# ------------------------------------------------------------------ planted mistakes
def _mutant(**overrides):
    ns = types.SimpleNamespace(**{k: getattr(REAL, k) for k in dir(REAL) if not k.startswith("__")})
    for k, v in overrides.items():
        setattr(ns, k, v)
    return ns


def _sal_interleaved_groups(K, Q, row_chunk=256):
    # wrong GQA convention: q head g reads KV head g % Hkv
    Hkv = K.shape[0]
    Hq = Q.shape[0]
    G = Hq // Hkv
    perm = np.array([h + Hkv * g for h in range(Hkv) for g in range(G)])
    return REAL.window_attention_saliency(K, Q[perm], row_chunk)


def _sal_no_causal(K, Q, row_chunk=256):
    Kf, Qf = REAL.bf16_to_f64(K), REAL.bf16_to_f64(Q)
    Hkv, T, d = Kf.shape
    G = Qf.shape[0] // Hkv
    W = Qf.shape[1]
    A = np.zeros((Hkv, T))
    for h in range(Hkv):
        s = Qf[h * G:(h + 1) * G].reshape(-1, d) @ Kf[h].T / math.sqrt(d)
        A[h] = softmax(s, axis=1).sum(axis=0) / G
    return A


def _sal_no_scale(K, Q, row_chunk=256):
    # logits without the 1/sqrt(d) scale
    return _scaled(K, Q, 1.0)


def _scaled(K, Q, scale):
    Kf, Qf = REAL.bf16_to_f64(K), REAL.bf16_to_f64(Q)
    Hkv, T, d = Kf.shape
    G, W = Qf.shape[0] // Hkv, Qf.shape[1]
    A = np.zeros((Hkv, T))
    j = np.arange(T)
    for h in range(Hkv):
        rows = Qf[h * G:(h + 1) * G].reshape(G * W, d)
        p = T - W + np.arange(G * W) % W
        s = rows @ Kf[h].T * scale
        s = np.where(j[None] <= p[:, None], s, -np.inf)
        A[h] = softmax(s, axis=1).sum(axis=0) / G
    return A


def _reuse_uncapped(c_prev, obs_sim, eta):
    c = np.asarray(c_prev, float).copy()
    t = len(c) - 1
    c[t] = 0.0
    if obs_sim is not None:
        c[:t] += eta * np.asarray(obs_sim, float)[:t]
    return c


def _reuse_no_reset(c_prev, obs_sim, eta):
    c = np.asarray(c_prev, float).copy()
    t = len(c) - 1
    if obs_sim is not None:
        for k in range(t):
            c[k] += min(1.0, eta * obs_sim[k])
    return c


def _utility_no_inner_clip(r, c, p):
    return REAL.clip(p.w_r * np.asarray(r, float) + p.w_c * np.log1p(np.asarray(c, float)), 0.0, p.s_max)


def _utility_log10(r, c, p):
    return REAL.clip(p.w_r * REAL.clip(np.asarray(r, float), p.r_min, p.r_max)
                     + p.w_c * np.log10(1 + np.asarray(c, float)), 0.0, p.s_max)


def _completion_wrong_sign(valid, gain, red, lam):
    return np.asarray(valid, float) + np.asarray(gain, float) + lam * np.asarray(red, float)


def _select_newer_wins(P, prunable, B):
    idx = np.nonzero(prunable)[0]
    order = np.lexsort((-idx, -P[idx]))
    return np.sort(idx[order[:B]])


def _budget_no_floor_one(N, mode, num=1, den=1, count=0):
    if N <= 0:
        return 0
    return min((num * N) // den if mode == "ratio" else count, N)


def _decode_interleaved(q, K, V):
    # wrong GQA convention: q head g reads KV head g % Hkv
    Hkv = K.shape[0]
    Hq = q.shape[0]
    G = Hq // Hkv
    inv = np.array([(g % Hkv) * G + g // Hkv for g in range(Hq)])
    out = REAL.decode_attention(q[np.argsort(inv)], K, V)
    return out[inv]


def _decode_no_scale(q, K, V):
    qf, Kf, Vf = REAL.bf16_to_f64(q), REAL.bf16_to_f64(K), REAL.bf16_to_f64(V)
    Hq, d = qf.shape
    G = Hq // Kf.shape[0]
    out = np.zeros((Hq, d))
    for g in range(Hq):
        out[g] = softmax(Kf[g // G] @ qf[g]) @ Vf[g // G]
    return out


def _decode_unnormalised(q, K, V):
    qf, Kf, Vf = REAL.bf16_to_f64(q), REAL.bf16_to_f64(K), REAL.bf16_to_f64(V)
    Hq, d = qf.shape
    G = Hq // Kf.shape[0]
    out = np.zeros((Hq, d))
    for g in range(Hq):
        s = Kf[g // G] @ qf[g] / math.sqrt(d)
        out[g] = np.exp(s - s.max()) @ Vf[g // G]
    return out


def _stats_keyed_previous_step(T_hat, step_id, prunable, chosen, n_steps):
    # keyed by step_id - 1: step 0's tokens wrap into the last step (totals unchanged)
    return REAL.step_statistics(T_hat, np.asarray(step_id) - 1, prunable, chosen, n_steps)


def _stats_max_over_all(T_hat, step_id, prunable, chosen, n_steps):
    # maximum taken over protected tokens of a step as well
    st = REAL.step_statistics(T_hat, step_id, prunable, chosen, n_steps)
    smax = np.zeros(n_steps)
    for i in range(len(T_hat)):
        k = int(step_id[i])
        if 0 <= k < n_steps:
            smax[k] = max(smax[k], T_hat[i])
    st["sal_max"] = smax
    return st


def _stats_count_protected(T_hat, step_id, prunable, chosen, n_steps):
    # counts every token of a step, protected ones included
    st = REAL.step_statistics(T_hat, step_id, prunable, chosen, n_steps)
    sid = np.asarray(step_id)
    st["count"] = np.array([int((sid == k).sum()) for k in range(n_steps)])
    return st


def _boundary_stats_on_raw(A_layers, step_id, prot, valid, gain, red, obs_sim, reuse_prev, p, budget_mode,
                           num=1, den=1, count=0):
    # per-step sums and maxima of the raw saliency T instead of the normalised T_hat
    out = REAL.stepkv_boundary(A_layers, step_id, prot, valid, gain, red, obs_sim, reuse_prev, p, budget_mode,
                               num, den, count)
    st = REAL.step_statistics(out["T"], step_id, ~np.asarray(prot).astype(bool), out["chosen"], len(valid))
    out.update({"step_" + k: v for k, v in st.items()})
    return out


def _mass_sum_over_group(q, K):
    # sum over the GQA group instead of the mean
    return REAL.decode_attention_mass(q, K) * (q.shape[0] // K.shape[0])


def _mass_no_scale(q, K):
    qf, Kf = REAL.bf16_to_f64(q), REAL.bf16_to_f64(K)
    G = qf.shape[0] // Kf.shape[0]
    A = np.zeros(Kf.shape[:2])
    for g in range(qf.shape[0]):
        A[g // G] += softmax(Kf[g // G] @ qf[g]) / G
    return A


def _mass_interleaved(q, K):
    # wrong GQA convention: q head g reads KV head g % Hkv
    Hkv = K.shape[0]
    G = q.shape[0] // Hkv
    perm = np.array([h + Hkv * g for h in range(Hkv) for g in range(G)])
    return REAL.decode_attention_mass(q[perm], K)


def _sim_dice(a, b):
    A, B = set(a), set(b)
    return 2 * len(A & B) / (len(A) + len(B)) if (A or B) else 0.0


def _signals_with(sim):
    def f(th, act, obs, k0=None):
        saved = REAL.cue_similarity
        REAL.cue_similarity = sim
        try:
            return saved.__globals__["step_signals"](th, act, obs, k0)
        finally:
            REAL.cue_similarity = saved
    return f


def _signals_mean_redundancy(th, act, obs, k0=None):
    gain, red, obs_sim = REAL.step_signals(th, act, obs, k0)
    n = len(obs)
    for k in range(0 if k0 is None else k0, n):
        red[k] = np.mean([REAL.cue_similarity(act[k], act[u]) for u in range(k)]) if k else 0.0
    return gain, red, obs_sim


def _signals_obs_only_gain(th, act, obs, k0=None):
    gain, red, obs_sim = REAL.step_signals(th, act, obs, k0)
    for k in range(0 if k0 is None else k0, len(obs)):
        gain[k] = 1.0 - max([REAL.cue_similarity(obs[k], obs[u]) for u in range(k)], default=0.0)
    return gain, red, obs_sim


def _lse_interleaved_groups(K, Q):
    # wrong GQA convention: q head g reads KV head g % Hkv
    Hkv = K.shape[0]
    order = np.concatenate([np.arange(g, Q.shape[0], Hkv) for g in range(Hkv)])
    out = np.empty((Q.shape[0], Q.shape[1]))
    out[order] = REAL.window_row_lse(K, Q[order])
    return out


def _lse_not_causal(K, Q):
    # every query row sees all T keys
    from scipy.special import logsumexp
    Kf, Qf = wl.bf16_bits_to_f32(K).astype(np.float64), wl.bf16_bits_to_f32(Q).astype(np.float64)
    G = Q.shape[0] // K.shape[0]
    return np.stack([logsumexp(Qf[g] @ Kf[g // G].T / math.sqrt(K.shape[2]), axis=1) for g in range(Q.shape[0])])


def _pool_window_shifted(a, k, mode="max"):
    # window [i - k//2 + 1, i + k//2 + 1]: off by one to the right
    b = np.concatenate([np.asarray(a, dtype=np.float64)[1:], [-np.inf if mode == "max" else np.nan]])
    return REAL.pool_tokens(b, k, mode)


def _pool_avg_counts_padding(a, k, mode="max"):
    out = REAL.pool_tokens(a, k, mode)
    if mode != "avg":
        return out
    a = np.asarray(a, dtype=np.float64)
    padded = np.concatenate([np.zeros(k // 2), a, np.zeros(k // 2)])
    return np.convolve(padded, np.ones(k) / k, mode="valid")


def _token_saliency_pool_after_mean(A_layers, pool=1, pool_mode="max"):
    T = REAL.token_saliency(A_layers)
    return REAL.pool_tokens(T, pool, pool_mode) if pool > 1 else T


@pytest.mark.parametrize("check, mutant", [
    (check_gqa_grouping, _mutant(window_attention_saliency=_sal_interleaved_groups)),
    (check_zero_keys_closed_form, _mutant(window_attention_saliency=_sal_no_causal)),
    (check_two_key_analytic, _mutant(window_attention_saliency=_sal_no_scale)),
    (check_reuse_table, _mutant(reuse_update=_reuse_uncapped)),
    (check_reuse_table, _mutant(reuse_update=_reuse_no_reset)),
    (check_step_utility_table, _mutant(step_utility=_utility_no_inner_clip)),
    (check_step_utility_table, _mutant(step_utility=_utility_log10)),
    (check_step_utility_table, _mutant(completion_score=_completion_wrong_sign)),
    (check_select_bruteforce, _mutant(select_top=_select_newer_wins)),
    (check_budget, _mutant(budget_tokens=_budget_no_floor_one)),
    (check_decode_gqa, _mutant(decode_attention=_decode_interleaved)),
    (check_decode_two_key_analytic, _mutant(decode_attention=_decode_no_scale)),
    (check_decode_identical_keys, _mutant(decode_attention=_decode_unnormalised)),
    (check_decode_bruteforce, _mutant(decode_attention=_decode_no_scale)),
    (check_step_statistics_table, _mutant(step_statistics=_stats_keyed_previous_step)),
    (check_step_statistics_table, _mutant(step_statistics=_stats_max_over_all)),
    (check_step_statistics_table, _mutant(step_statistics=_stats_count_protected)),
    (check_boundary_step_statistics, _mutant(stepkv_boundary=_boundary_stats_on_raw)),
    (check_mass_sums, _mutant(decode_attention_mass=_mass_sum_over_group)),
    (check_mass_two_key_analytic, _mutant(decode_attention_mass=_mass_no_scale)),
    (check_mass_bruteforce, _mutant(decode_attention_mass=_mass_no_scale)),
    (check_mass_gqa, _mutant(decode_attention_mass=_mass_interleaved)),
    (check_cue_similarity_cases, _mutant(cue_similarity=_sim_dice)),
    (check_step_signals_table, _mutant(step_signals=_signals_with(_sim_dice))),
    (check_step_signals_table, _mutant(step_signals=_signals_mean_redundancy)),
    (check_step_signals_table, _mutant(step_signals=_signals_obs_only_gain)),
    (check_pool_table, _mutant(pool_tokens=_pool_window_shifted)),
    (check_pool_max_library, _mutant(pool_tokens=_pool_window_shifted)),
    (check_pool_table, _mutant(pool_tokens=_pool_avg_counts_padding)),
    (check_pool_avg_convolution, _mutant(pool_tokens=_pool_avg_counts_padding)),
    (check_pool_before_mean, _mutant(token_saliency=_token_saliency_pool_after_mean)),
    (check_lse_logsumexp, _mutant(window_row_lse=_lse_interleaved_groups)),
    (check_lse_rebuilds_saliency, _mutant(window_row_lse=_lse_interleaved_groups)),
    (check_lse_zero_keys, _mutant(window_row_lse=_lse_not_causal)),
])
def test_planted_mistake_is_caught(check, mutant):
    with pytest.raises(AssertionError):
        check(mutant)
