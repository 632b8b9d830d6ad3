"""GPU parity of every stage against the CPU oracle, through the C ABI (libstepkv.so).

Sizes span several 128-key tiles with ragged tails, row groups above 256 query rows, windows split
over row groups, d = 64 and 128, GQA groups 1/2/4/5, the paper's seeds (233, 42, 3407) and the
full 32K-token, 32-layer workload the benchmark times.
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


def _rand_bits(rng, shape, scale=1.0):
    return wl.f32_to_bf16_bits(rng.standard_normal(shape).astype(np.float32) * np.float32(scale))


# ------------------------------------------------------------------------------------ stage 1
SCORE_CASES = [
    # Hkv, G, d, T, W, n_layers
    (2, 4, 64, 2048, 32, 1),     # tiny workload shape
    (8, 4, 128, 4100, 64, 2),    # ragged T, one row group of 256
    (2, 5, 128, 1000, 128, 1),   # 640 query rows -> 3 row groups
    (1, 1, 128, 300, 1, 1),      # single query (textbook softmax case)
    (2, 2, 64, 130, 7, 3),       # W not a multiple of 8
    (1, 2, 128, 700, 300, 1),    # window split over two row groups
    (4, 1, 64, 64, 64, 1),       # W = T, T below one tile
    (2, 4, 128, 127, 5, 1),
    (1, 8, 128, 513, 33, 1),     # 8 heads x 40 padded rows = 320 rows -> 2 row groups
]


@pytest.mark.parametrize("Hkv,G,d,T,W,nl", SCORE_CASES)
def test_score_matches_oracle(B, Hkv, G, d, T, W, nl):
    import torch
    rng = np.random.default_rng(1000 + T + W)
    Ks = [_rand_bits(rng, (Hkv, T, d)) for _ in range(nl)]
    Qs = [_rand_bits(rng, (Hkv * G, W, d)) for _ in range(nl)]
    st = B.new_status()
    sal = B.stepkv_score([TL.bf16_dev(k) for k in Ks], [TL.bf16_dev(q) for q in Qs], T, status=st)
    torch.cuda.synchronize()
    assert st.item() == 0
    g = sal.cpu().numpy()
    for l in range(nl):
        ref = O.window_attention_saliency(Ks[l], Qs[l])
        TL.assert_close(g[l], ref, f"sal layer {l}")
        assert np.allclose(g[l].sum(axis=1), W, rtol=1e-4)


@pytest.mark.parametrize("Hkv,G,d,T,W,nl", SCORE_CASES + [(1, 4, 128, 2500, 512, 1), (1, 5, 128, 3000, 1024, 1)])
def test_score_with_prefill_lse_matches_oracle(B, Hkv, G, d, T, W, nl):
    """stepkv_score_lse: the rows' log-sum-exp comes from the caller (the oracle's, rounded to fp32, as
    a prefill attention kernel would report it) and only the second pass runs."""
    import torch
    rng = np.random.default_rng(2000 + T + W)
    Ks = [_rand_bits(rng, (Hkv, T, d)) for _ in range(nl)]
    Qs = [_rand_bits(rng, (Hkv * G, W, d)) for _ in range(nl)]
    lse = [torch.from_numpy(O.window_row_lse(k, q).astype(np.float32)).cuda() for k, q in zip(Ks, Qs)]
    st = B.new_status()
    sal = B.stepkv_score([TL.bf16_dev(k) for k in Ks], [TL.bf16_dev(q) for q in Qs], T, status=st, lse=lse)
    torch.cuda.synchronize()
    assert st.item() == 0
    g = sal.cpu().numpy()
    for l in range(nl):
        TL.assert_close(g[l], O.window_attention_saliency(Ks[l], Qs[l]), f"sal layer {l}")


def test_compress_with_prefill_lse(B):
    """The fused pass with each saliency layer's row log-sum-exp given (stepkv_problem_t.sal_lse): pass 1
    is skipped and every output matches the oracle."""
    import torch
    tr = wl.custom(83, L=4, Hq=16, Hkv=4, d=128, T=6000, W=64, n_steps=12, budget=wl.Budget.ratio(1, 8))
    g = TL.GpuTraj(tr)
    prob = g.problem()
    prob.sal_lse = [torch.from_numpy(O.window_row_lse(tr.keys(l), tr.queries(l)).astype(np.float32)).cuda()
                    for l in tr.sal_layer_ids()]
    prob.refresh()
    p = B.Params()
    st = B.stepkv_compress([prob], p)
    torch.cuda.synchronize()
    assert st.item() == 0
    TL.check_select_outputs(g, TL.run_oracle(tr, TL.oracle_params(p)))
    n = int(g.out.n_kept.item())
    kt = g.out.kept_idx[:n].long()
    for l in range(tr.shape.L):
        assert torch.equal(g.K_out[l][:, :n], g.K[l].index_select(1, kt))


def test_score_with_prefill_lse_uses_it(B):
    """An lse raised by delta for one query head scales that head's share of the saliency by exp(-delta):
    the kernel takes the caller's statistics instead of recomputing them."""
    import torch
    rng = np.random.default_rng(17)
    Hkv, G, d, T, W = 2, 4, 128, 3000, 64
    K, Q = _rand_bits(rng, (Hkv, T, d)), _rand_bits(rng, (Hkv * G, W, d))
    lse = O.window_row_lse(K, Q)
    delta = 0.7
    lse_shift = lse.copy()
    lse_shift[5] += delta  # query head 5 = KV head 1, group member 1
    sal = B.stepkv_score([TL.bf16_dev(K)], [TL.bf16_dev(Q)], T,
                         lse=[torch.from_numpy(lse_shift.astype(np.float32)).cuda()])
    torch.cuda.synchronize()
    # the reference: head 5's rows weighted by exp(-delta) (the saliency rebuilt from the oracle's rows)
    Kf, Qf = wl.bf16_bits_to_f32(K).astype(np.float64), wl.bf16_bits_to_f32(Q).astype(np.float64)
    ref = np.zeros((Hkv, T))
    for gq in range(Hkv * G):
        for w in range(W):
            vis = T - W + w + 1
            s = Qf[gq, w] @ Kf[gq // G, :vis].T / np.sqrt(d)
            ref[gq // G, :vis] += np.exp(s - lse_shift[gq, w]) / G
    TL.assert_close(sal.cpu().numpy()[0], ref, "sal with a shifted lse")
    assert abs(ref[1].sum() - (W * (G - 1) + W * np.exp(-delta)) / G) < 1e-6 * W


# Observation-length windows (the queries are a whole last Observation, hundreds to 4096 tokens): the
# window is split over up to 16 row groups per query head, GQA 4 and 5.
LONG_WINDOW_CASES = [
    # Hkv, G, d, T, W
    (1, 4, 128, 2500, 512),
    (1, 5, 128, 3000, 1024),
    pytest.param(1, 4, 128, 5000, 4096, marks=pytest.mark.slow),
    pytest.param(1, 5, 128, 4300, 4096, marks=pytest.mark.slow),
]


@pytest.mark.parametrize("Hkv,G,d,T,W", LONG_WINDOW_CASES)
def test_score_observation_length_window(B, Hkv, G, d, T, W):
    import torch
    rng = np.random.default_rng(2000 + T + W + G)
    K = _rand_bits(rng, (Hkv, T, d))
    Q = _rand_bits(rng, (Hkv * G, W, d))
    st = B.new_status()
    sal = B.stepkv_score([TL.bf16_dev(K)], [TL.bf16_dev(Q)], T, status=st)
    torch.cuda.synchronize()
    assert st.item() == 0
    g = sal[0].cpu().numpy()
    TL.assert_close(g, O.window_attention_saliency(K, Q), f"sal W={W}")
    assert np.allclose(g.sum(axis=1), W, rtol=1e-4)


def test_compress_observation_window(B):
    """The fused pass with a 1024-token window (fixed-point accumulation over 16 row groups per pair)."""
    import torch
    tr = wl.custom(61, L=3, Hq=8, Hkv=2, d=128, T=3000, W=1024, n_steps=3, budget=wl.Budget.ratio(1, 4))
    assert tr.step_id[-1] == tr.n_steps - 1 and (tr.step_id[-tr.shape.W:] == tr.n_steps - 1).all()
    g = TL.GpuTraj(tr)
    prob = g.problem()
    st = B.stepkv_compress([prob], B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    TL.check_select_outputs(g, TL.run_oracle(tr, O.Params()))


@pytest.mark.slow
def test_score_observation_prefill_full_size_sampled(B):
    """The 32K Llama-shaped trajectory with its whole last Observation (2048 tokens, 8192 query rows per
    KV head) as the window, in the launch the fused pass makes (all 3 saliency layers): one sampled
    (layer, KV head) pair is computed by the oracle and compared over all 32768 keys; every pair's
    masses must sum to W (each query row's softmax sums to one)."""
    import torch
    tr = wl.observation_prefill("llama8b_32k", 2048)
    s = tr.shape
    Ks = [tr.keys(l) for l in tr.sal_layer_ids()]
    Qs = [tr.queries(l) for l in tr.sal_layer_ids()]
    st = B.new_status()
    sal = B.stepkv_score([TL.bf16_dev(k) for k in Ks], [TL.bf16_dev(q) for q in Qs], s.T, status=st)
    torch.cuda.synchronize()
    assert st.item() == 0
    g = sal.cpu().numpy()
    assert np.allclose(g.sum(axis=2), s.W, rtol=1e-4)
    li, h = 1, 5
    ref = O.window_attention_saliency(Ks[li][h:h + 1], Qs[li][h * s.G:(h + 1) * s.G])[0]
    TL.assert_close(g[li, h], ref, "sal full-size observation window, layer 1 head 5")


# Table 2 and Table 3 ablations as oracle-checked modes of the fused pass: no redundancy penalty (lambda = 0),
# no reuse credit (eta = 0), step utility alone (alpha = 0) and token saliency alone (beta = 0), plus the
# un-normalised saliency.
ABLATIONS = [
    {"lam": 0.0}, {"eta": 0.0}, {"alpha": 0.0, "beta": 1.0}, {"alpha": 1.0, "beta": 0.0},
    {"alpha": 0.5, "beta": 0.5, "sal_norm": 1},
]


@pytest.mark.parametrize("ablation", ABLATIONS, ids=lambda a: "-".join(f"{k}{v}" for k, v in a.items()))
def test_compress_ablation_modes(B, ablation):
    import torch
    tr = wl.custom(81, L=4, Hq=16, Hkv=4, d=128, T=5000, W=64, n_steps=12, budget=wl.Budget.ratio(1, 8))
    p = B.Params()
    for k, v in ablation.items():
        setattr(p, k, v)
    g = TL.GpuTraj(tr)
    prob = g.problem()
    st = B.stepkv_compress([prob], p)
    torch.cuda.synchronize()
    assert st.item() == 0
    out = TL.run_oracle(tr, TL.oracle_params(p))
    TL.check_select_outputs(g, out)
    n = int(g.out.n_kept.item())
    kt = g.out.kept_idx[:n].long()
    for l in range(tr.shape.L):
        assert torch.equal(g.K_out[l][:, :n], g.K[l].index_select(1, kt))
        assert torch.equal(g.V_out[l][:, :n], g.V[l].index_select(1, kt))


def test_score_capacity_head_stride(B):
    """K rows live in a larger capacity buffer ([Hkv, cap, d] with cap > T)."""
    import torch
    rng = np.random.default_rng(7)
    Hkv, G, d, T, W, cap = 2, 4, 128, 1500, 64, 2048
    Kfull = _rand_bits(rng, (Hkv, cap, d))
    Q = _rand_bits(rng, (Hkv * G, W, d))
    Kd = TL.bf16_dev(Kfull)[:, :T]  # strided view: head stride cap*d
    sal = B.stepkv_score([Kd], [TL.bf16_dev(Q)], T)
    torch.cuda.synchronize()
    ref = O.window_attention_saliency(np.ascontiguousarray(Kfull[:, :T]), Q)
    TL.assert_close(sal[0].cpu().numpy(), ref, "sal (capacity layout)")


def test_score_outlier_channels(B):
    """Keys with 4 channels scaled x8 (the ragged-batch workload's outliers): wider logit range."""
    import torch
    tr = wl.custom(11, L=3, Hq=32, Hkv=8, d=128, T=3000, W=64, n_steps=6, outlier_channels=4)
    Ks = [tr.keys(l) for l in tr.sal_layer_ids()]
    Qs = [tr.queries(l) for l in tr.sal_layer_ids()]
    sal = B.stepkv_score([TL.bf16_dev(k) for k in Ks], [TL.bf16_dev(q) for q in Qs], tr.T)
    torch.cuda.synchronize()
    for l in range(3):
        TL.assert_close(sal[l].cpu().numpy(), O.window_attention_saliency(Ks[l], Qs[l]), "sal outliers")


def test_score_logit_jumps(B):
    """Logits that jump far above everything a row has seen earlier in its key range: the last 32 keys
    of every 128 sit 4.5 higher in every channel along the queries' common direction (about 2^73 above
    the rest after the log2(e)/sqrt(d) scale), and the last 32 of every 512 sit 9 higher (2^147: a sum
    taken against the earlier maximum overflows fp32).  Masses below 1e-30 are compared absolutely (the
    kernel's exponential flushes results below 2^-126 to zero)."""
    import torch
    rng = np.random.default_rng(77)
    Hkv, G, d, T, W = 2, 2, 128, 2000, 16
    j = np.arange(T)
    t = np.where(j % 512 >= 480, 9.0, np.where(j % 128 >= 96, 4.5, 0.0)).astype(np.float32)
    K = wl.f32_to_bf16_bits(rng.standard_normal((Hkv, T, d)).astype(np.float32) * 0.25 + t[None, :, None])
    Q = wl.f32_to_bf16_bits(rng.standard_normal((Hkv * G, W, d)).astype(np.float32) * 0.25 + 1.0)
    st = B.new_status()
    sal = B.stepkv_score([TL.bf16_dev(K)], [TL.bf16_dev(Q)], T, status=st)
    torch.cuda.synchronize()
    assert st.item() == 0
    g = sal[0].cpu().numpy()
    ref = O.window_attention_saliency(K, Q)
    assert np.all(np.isfinite(g))
    TL.assert_close(g, ref, "sal (logit jumps)", floor=1e-30)
    assert np.allclose(g.sum(axis=1), W, rtol=1e-4)


# ------------------------------------------------------------------------------------ stages 2-4
def _select_case(B, tr, p, sal_fp32, kept_cap=None):
    import torch
    g = TL.GpuTraj.__new__(TL.GpuTraj)
    g.tr = tr
    g.step_id = torch.from_numpy(tr.step_id).cuda()
    g.prot = torch.from_numpy(tr.prot).cuda()
    g.valid = torch.from_numpy(tr.valid).cuda()
    g.gain = torch.from_numpy(tr.gain).cuda()
    g.red = torch.from_numpy(tr.red).cuda()
    g.obs_sim = torch.from_numpy(tr.obs_sim).cuda()
    g.reuse_in = torch.from_numpy(tr.reuse).cuda()
    g.reuse_out = torch.empty_like(g.reuse_in)
    cap = kept_cap if kept_cap is not None else tr.T
    g.out = B.SelectOutputs.allocate(tr.T, tr.n_steps, cap, "cuda")
    st = B.new_status()
    b = tr.budget
    bud = B.budget_ratio(b.num, b.den) if b.mode == "ratio" else B.budget_count(b.count)
    B.stepkv_select(torch.from_numpy(sal_fp32).cuda(), g.step_id, g.prot, g.steps(), p, bud, g.out, status=st)
    torch.cuda.synchronize()
    A = [sal_fp32[i].astype(np.float64) for i in range(sal_fp32.shape[0])]
    out = O.stepkv_boundary([a[None] for a in A], tr.step_id, tr.prot, tr.valid, tr.gain, tr.red, tr.obs_sim,
                            tr.reuse, TL.oracle_params(p), b.mode, b.num, b.den, b.count)
    return g, out, int(st.item())


@pytest.mark.parametrize("seed", [0, 233, 42, 3407])
def test_select_matches_oracle(B, seed):
    tr = wl.tiny(seed)
    Ks = [tr.keys(l) for l in tr.sal_layer_ids()]
    Qs = [tr.queries(l) for l in tr.sal_layer_ids()]
    sal = np.concatenate([O.window_attention_saliency(k, q) for k, q in zip(Ks, Qs)]).astype(np.float32)
    g, out, st = _select_case(B, tr, B.Params(), sal)
    assert st == 0
    TL.check_select_outputs(g, out)


@pytest.mark.parametrize("T", [2047, 2048, 2049, 2065])
def test_select_single_cta_cluster_boundary(B, T):
    """Up to 2048 tokens one CTA selects, above that an 8-CTA cluster: both sides of the switch."""
    tr = wl.custom(17, L=1, Hq=4, Hkv=1, d=64, T=T, W=16, n_steps=7, budget=wl.Budget.ratio(1, 4))
    rng = np.random.default_rng(T)
    sal = (rng.random((2, tr.T)) * 2).astype(np.float32)
    g, out, st = _select_case(B, tr, B.Params(), sal)
    assert st == 0
    TL.check_select_outputs(g, out)


@pytest.mark.parametrize("budget", [wl.Budget.ratio(1, 10), wl.Budget.ratio(1, 2), wl.Budget.fixed(1),
                                    wl.Budget.fixed(5000), wl.Budget.ratio(1, 1), wl.Budget.fixed(0)])
def test_select_budgets(B, budget):
    tr = wl.custom(5, L=1, Hq=4, Hkv=1, d=64, T=4000, W=16, n_steps=9, budget=budget)
    rng = np.random.default_rng(3)
    sal = (rng.random((2, tr.T)) * 3).astype(np.float32)
    g, out, st = _select_case(B, tr, B.Params(), sal)
    assert st == 0
    TL.check_select_outputs(g, out)


@pytest.mark.parametrize("levels", [2, 7, 150, 200, 1000])
def test_select_exact_on_shared_fp32_priorities(B, levels):
    """alpha=1, beta=0, no normalisation, one saliency row: the kernel ranks exactly the fp32 values
    it is given, so its retained set must equal the oracle's ranking of the same values bit for bit,
    ties (few distinct levels) included.  ~100-130 tokens per level (150 and 200 levels over 20000
    tokens) put the threshold bin on both sides of the 128 candidates the value-bin path resolves
    directly; 2 and 7 levels take the radix fallback."""
    import torch
    T = 20000
    tr = wl.custom(9, L=1, Hq=1, Hkv=1, d=64, T=T, W=8, n_steps=12, budget=wl.Budget.ratio(3, 10))
    rng = np.random.default_rng(levels)
    sal = (rng.integers(0, levels, (1, T)) / levels).astype(np.float32)
    p = B.Params(alpha=1.0, beta=0.0, sal_norm=B.NORM_NONE)
    g, out, st = _select_case(B, tr, p, sal)
    assert st == 0
    n = int(g.out.n_kept.item())
    gk = g.out.kept_idx[:n].cpu().numpy()
    prunable = ~tr.prot.astype(bool)
    Bt = O.budget_tokens(int(prunable.sum()), "ratio", 3, 10)
    exp = O.kept_indices(tr.prot, O.select_top(sal[0].astype(np.float64), prunable, Bt))
    assert np.array_equal(gk, exp)
    assert np.array_equal(g.out.step_kept.cpu().numpy(), out["step_kept"])


@pytest.mark.parametrize("pool, mode, T", [(3, 0, 9000), (7, 0, 9000), (7, 1, 9000), (63, 1, 9000), (31, 0, 9000),
                                           (5, 1, 1500)])
def test_select_snapkv_pooling(B, pool, mode, T):
    """SnapKV-style estimator: every saliency row pooled over `pool` tokens (max or in-range mean) before
    the mean over rows, then Eqs. 2-5 and the selection, against the oracle (windows clipped at both ends;
    T = 1500 takes the single-CTA selection)."""
    tr = wl.custom(11 + pool, L=1, Hq=8, Hkv=2, d=64, T=T, W=16, n_steps=10, budget=wl.Budget.ratio(1, 5))
    rng = np.random.default_rng(pool * 10 + mode)
    sal = (rng.random((6, tr.T)) ** 3).astype(np.float32)
    p = B.Params(sal_pool=pool, sal_pool_mode=mode)
    g, out, st = _select_case(B, tr, p, sal)
    assert st == 0
    TL.check_select_outputs(g, out)


@pytest.mark.parametrize("pool, mode, W, lse", [(7, 0, 64, False), (5, 1, 64, True), (3, 0, 128, False)])
def test_compress_with_snapkv_pooling(B, pool, mode, W, lse):
    """The fused pass with a pooled token saliency: the saliency rows are written and pooled per
    trajectory (with and without the prefill's row statistics; W = 128 at GQA 4 takes two row groups)."""
    import torch
    tr = wl.custom(60 + pool, L=4, Hq=16, Hkv=4, d=128, T=5000, W=W, n_steps=12, budget=wl.Budget.ratio(1, 8))
    g = TL.GpuTraj(tr)
    prob = g.problem()
    if lse:
        prob.sal_lse = [torch.from_numpy(O.window_row_lse(tr.keys(l), tr.queries(l)).astype(np.float32)).cuda()
                        for l in tr.sal_layer_ids()]
        prob.refresh()
    p = B.Params(sal_pool=pool, sal_pool_mode=mode)
    st = B.stepkv_compress([prob], p)
    torch.cuda.synchronize()
    assert st.item() == 0
    TL.check_select_outputs(g, TL.run_oracle(tr, TL.oracle_params(p)))
    n = int(g.out.n_kept.item())
    kt = g.out.kept_idx[:n].long()
    assert torch.equal(g.K_out[0][:, :n], g.K[0].index_select(1, kt))


def test_select_large_T(B):
    """T = 200000 (beyond 8 x 16K): every CTA of the cluster holds ~25K tokens."""
    T = 200000
    tr = wl.custom(21, L=1, Hq=8, Hkv=2, d=64, T=T, W=64, n_steps=150, budget=wl.Budget.fixed(8192))
    rng = np.random.default_rng(21)
    sal = rng.random((6, T)).astype(np.float32) ** 4
    g, out, st = _select_case(B, tr, B.Params(), sal)
    assert st == 0
    TL.check_select_outputs(g, out)


@pytest.mark.parametrize("n_steps", [2048, 2600])
def test_select_many_steps(B, n_steps):
    """Thousands of reasoning steps (a few tokens each): per-step statistics, S_k and the selection."""
    T = 24000
    tr = wl.custom(31 + n_steps, L=1, Hq=8, Hkv=2, d=64, T=T, W=32, n_steps=n_steps, budget=wl.Budget.ratio(1, 6))
    rng = np.random.default_rng(n_steps)
    sal = rng.random((2, T)).astype(np.float32) ** 3
    g, out, st = _select_case(B, tr, B.Params(), sal)
    assert st == 0
    TL.check_select_outputs(g, out)


def test_select_reuse_in_place(B):
    """reuse_out may alias reuse_in (the caller keeps one c_k array across boundaries)."""
    import torch
    tr = wl.custom(6, L=1, Hq=4, Hkv=1, d=64, T=5000, W=16, n_steps=30)
    rng = np.random.default_rng(6)
    sal = (rng.random((2, tr.T)) * 3).astype(np.float32)
    c = torch.from_numpy(tr.reuse.copy()).cuda()
    steps = B.StepSignals(*(torch.from_numpy(x).cuda() for x in (tr.valid, tr.gain, tr.red)), c,
                          torch.from_numpy(tr.obs_sim).cuda(), c)
    out = B.SelectOutputs.allocate(tr.T, tr.n_steps, tr.T, "cuda")
    st = B.new_status()
    B.stepkv_select(torch.from_numpy(sal).cuda(), torch.from_numpy(tr.step_id).cuda(), torch.from_numpy(tr.prot).cuda(),
                    steps, B.Params(), B.budget_ratio(1, 5), out, status=st)
    torch.cuda.synchronize()
    assert st.item() == 0
    exp = O.reuse_update(tr.reuse, tr.obs_sim, 1.5)
    TL.assert_close(c.cpu().numpy(), exp, "c_k in place", floor=1e-6)
    p = O.Params()
    S = O.step_utility(O.completion_score(tr.valid, tr.gain, tr.red, p.lam), exp, p)
    TL.assert_close(out.step_util.cpu().numpy(), S, "S_k", floor=1e-6)


def test_select_bad_step_id_sets_edata(B):
    tr = wl.custom(4, L=1, Hq=2, Hkv=1, d=64, T=600, W=8, n_steps=3)
    tr.step_id = tr.step_id.copy()
    assert tr.prot[300] == 0
    tr.step_id[300] = 3  # == n_steps: out of range
    g, _, st = _select_case_status(B, tr, np.ones((1, tr.T), np.float32))
    assert st == B.STEPKV_EDATA
    assert int(g.out.n_kept.item()) == 0


def _select_case_status(B, tr, sal):
    import torch
    g = TL.GpuTraj.__new__(TL.GpuTraj)
    g.tr = tr
    step_id = torch.from_numpy(tr.step_id).cuda()
    prot = torch.from_numpy(tr.prot).cuda()
    steps = B.StepSignals(*(torch.from_numpy(a).cuda() for a in (tr.valid, tr.gain, tr.red, tr.reuse)))
    g.out = B.SelectOutputs.allocate(tr.T, tr.n_steps, tr.T, "cuda")
    st = B.new_status()
    B.stepkv_select(torch.from_numpy(sal).cuda(), step_id, prot, steps, B.Params(), B.budget_ratio(1, 2), g.out,
                    status=st)
    torch.cuda.synchronize()
    return g, None, int(st.item())


# ------------------------------------------------------------------------------------ stage 5
@pytest.mark.parametrize("d", [64, 96, 128])
def test_compact_bit_exact(B, d):
    import torch
    rng = np.random.default_rng(d)
    L, Hkv, T, cap = 3, 4, 3001, 1200
    Kin = [_rand_bits(rng, (Hkv, T, d)) for _ in range(L)]
    Vin = [_rand_bits(rng, (Hkv, T, d)) for _ in range(L)]
    kept = np.sort(rng.choice(T, 1111, replace=False)).astype(np.int32)
    step_in = rng.integers(-1, 50, T).astype(np.int32)
    pos_in = (np.arange(T) * 3 + 7).astype(np.int32)
    Kout = [torch.zeros((Hkv, cap, d), dtype=torch.bfloat16, device="cuda") for _ in range(L)]
    Vout = [torch.zeros((Hkv, cap, d), dtype=torch.bfloat16, device="cuda") for _ in range(L)]
    kd = torch.zeros(cap, dtype=torch.int32, device="cuda")
    kd[:len(kept)] = torch.from_numpy(kept).cuda()
    nk = torch.tensor([len(kept)], dtype=torch.int32, device="cuda")
    so = torch.full((cap,), -9, dtype=torch.int32, device="cuda")
    po = torch.full((cap,), -9, dtype=torch.int32, device="cuda")
    st = B.new_status()
    B.stepkv_compact([TL.bf16_dev(k) for k in Kin], [TL.bf16_dev(v) for v in Vin], T, kd, nk, cap, Kout, Vout,
                     torch.from_numpy(step_in).cuda(), torch.from_numpy(pos_in).cuda(), so, po, status=st)
    torch.cuda.synchronize()
    assert st.item() == 0
    for l in range(L):
        assert np.array_equal(TL.bits_of(Kout[l])[:, :len(kept)], O.compact_rows(Kin[l], kept))
        assert np.array_equal(TL.bits_of(Vout[l])[:, :len(kept)], O.compact_rows(Vin[l], kept))
        assert np.all(TL.bits_of(Kout[l])[:, len(kept):] == 0)  # rows past n_kept untouched
    assert np.array_equal(so.cpu().numpy()[:len(kept)], step_in[kept])
    assert np.array_equal(po.cpu().numpy()[:len(kept)], pos_in[kept])
    assert np.all(so.cpu().numpy()[len(kept):] == -9)


def test_compact_rejects_overflow_on_device(B):
    import torch
    T, cap = 100, 10
    K = [torch.zeros((1, T, 64), dtype=torch.bfloat16, device="cuda")]
    Ko = [torch.zeros((1, cap, 64), dtype=torch.bfloat16, device="cuda")]
    kd = torch.arange(cap, dtype=torch.int32, device="cuda")
    nk = torch.tensor([cap + 1], dtype=torch.int32, device="cuda")
    st = B.new_status()
    B.stepkv_compact(K, None, T, kd, nk, cap, Ko, None, status=st)
    torch.cuda.synchronize()
    assert st.item() == B.STEPKV_ENOSPACE


# ------------------------------------------------------------------------------------ fused pass
def _compress_and_check(B, tr, p=None, layers_check=None, kept_cap=None):
    import torch
    p = p or B.Params()
    g = TL.GpuTraj(tr, kept_cap=kept_cap)
    prob = g.problem()
    st = B.stepkv_compress([prob], p)
    torch.cuda.synchronize()
    assert st.item() == 0, st.item()
    out = TL.run_oracle(tr, TL.oracle_params(p))
    swaps = TL.check_select_outputs(g, out)
    n = int(g.out.n_kept.item())
    gk = g.out.kept_idx[:n].cpu().numpy()
    for l in (layers_check if layers_check is not None else range(tr.shape.L)):
        assert np.array_equal(TL.bits_of(g.K_out[l])[:, :n], O.compact_rows(tr.keys(l), gk))
        assert np.array_equal(TL.bits_of(g.V_out[l])[:, :n], O.compact_rows(tr.values(l), gk))
    assert np.array_equal(g.step_id_out[:n].cpu().numpy(), tr.step_id[gk])
    assert np.array_equal(g.pos_out[:n].cpu().numpy(), tr.pos[gk])
    return g, out, swaps


@pytest.mark.parametrize("seed", [0, 233, 42, 3407])
def test_compress_tiny(B, seed):
    _compress_and_check(B, wl.tiny(seed))


def test_compress_medium_gqa5_w128(B):
    tr = wl.custom(77, L=5, Hq=10, Hkv=2, d=128, T=6000, W=128, n_steps=14, budget=wl.Budget.fixed(700))
    _compress_and_check(B, tr)


def test_compress_llama_shape_short(B):
    tr = wl.llama8b_32k(seed=5, T=8192, L=4)
    _compress_and_check(B, tr)


def test_compress_batched_ragged(B):
    import torch
    trs = [wl.custom(100 + i, L=3, Hq=8, Hkv=2, d=128, T=T, W=32, n_steps=5 + i, budget=wl.Budget.ratio(1, 5))
           for i, T in enumerate((1700, 2600, 999))]
    gs = [TL.GpuTraj(tr) for tr in trs]
    probs = [g.problem() for g in gs]
    st = B.stepkv_compress(probs, B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    for g, tr in zip(gs, trs):
        out = TL.run_oracle(tr, TL.oracle_params(B.Params()))
        TL.check_select_outputs(g, out)
        n = int(g.out.n_kept.item())
        gk = g.out.kept_idx[:n].cpu().numpy()
        assert np.array_equal(TL.bits_of(g.K_out[0])[:, :n], O.compact_rows(tr.keys(0), gk))


def test_compress_batched_mixed_prefill_lse(B):
    """Four ragged trajectories in one call, two with the prefill's row log-sum-exp and two without: the
    saliency batches split by mode (one launch may not mix them) and every trajectory matches the oracle."""
    import torch
    trs = [wl.custom(120 + i, L=3, Hq=8, Hkv=2, d=128, T=T, W=32, n_steps=5 + i, budget=wl.Budget.ratio(1, 5))
           for i, T in enumerate((1700, 2600, 999, 3100))]
    gs = [TL.GpuTraj(tr) for tr in trs]
    probs = [g.problem() for g in gs]
    for i in (0, 1):
        tr = trs[i]
        probs[i].sal_lse = [torch.from_numpy(O.window_row_lse(tr.keys(l), tr.queries(l)).astype(np.float32)).cuda()
                            for l in tr.sal_layer_ids()]
        probs[i].refresh()
    st = B.stepkv_compress(probs, B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    for g, tr in zip(gs, trs):
        TL.check_select_outputs(g, TL.run_oracle(tr, TL.oracle_params(B.Params())))


@pytest.mark.parametrize("Hq,Hkv,W", [(10, 2, 128), (4, 2, 300)])
def test_compress_batched_row_groups(B, Hq, Hkv, W):
    """Short trajectories whose query rows need several row groups (GQA 5 x W 128 = 640 rows; a
    300-row window split over two groups) share one saliency launch."""
    import torch
    trs = [wl.custom(500 + i + W, L=2, Hq=Hq, Hkv=Hkv, d=128, T=T, W=W, n_steps=4 + i, budget=wl.Budget.ratio(1, 3))
           for i, T in enumerate((700, 1300, 2100))]
    gs = [TL.GpuTraj(tr) for tr in trs]
    st = B.stepkv_compress([g.problem() for g in gs], B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    for g, tr in zip(gs, trs):
        TL.check_select_outputs(g, TL.run_oracle(tr, TL.oracle_params(B.Params())))


def test_compress_twenty_trajectories_mixed_in_place(B):
    """20 trajectories in one call (more than one selection launch of 16 and more than one compaction
    launch), every fourth compacted in place: each matches the oracle."""
    import torch
    trs = [wl.custom(600 + i, L=2, Hq=4, Hkv=2, d=64, T=400 + 37 * i, W=16, n_steps=3 + i % 4,
                     budget=wl.Budget.ratio(1, 5)) for i in range(20)]
    gs = [TL.GpuTraj(tr) for tr in trs]
    probs = []
    src = []
    for i, (g, tr) in enumerate(zip(gs, trs)):
        prob = g.problem()
        if i % 4 == 3:
            # in place: the outputs are the inputs (rows [0, n_kept) end up holding the retained set)
            src.append(([TL.bits_of(k) for k in g.K], [TL.bits_of(v) for v in g.V]))
            prob = B.Problem(g.K, g.V, g.Q, tr.T, g.step_id, g.prot, g.steps(), g.budget(), g.K, g.V, g.out,
                             pos_in=g.pos, step_id_out=g.step_id_out, pos_out=g.pos_out)
        else:
            src.append(None)
        probs.append(prob)
    st = B.stepkv_compress(probs, B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    for g, tr, sv in zip(gs, trs, src):
        out = TL.run_oracle(tr, TL.oracle_params(B.Params()))
        TL.check_select_outputs(g, out)
        n = int(g.out.n_kept.item())
        gk = g.out.kept_idx[:n].cpu().numpy().astype(np.int64)
        if sv is None:
            assert np.array_equal(TL.bits_of(g.K_out[1])[:, :n], O.compact_rows(tr.keys(1), gk))
        else:
            slot_of_pos = {int(x): j for j, x in enumerate(tr.pos)}
            srcs = np.array([slot_of_pos[int(x)] for x in g.pos_out[:n].cpu().numpy()], np.int64)
            assert np.array_equal(np.sort(srcs), gk)
            assert np.array_equal(TL.bits_of(g.K[1])[:, :n], sv[0][1][:, srcs])
            assert np.array_equal(TL.bits_of(g.V[0])[:, :n], sv[1][0][:, srcs])


@pytest.mark.parametrize("T,num,den,all_prot", [(20000, 1, 2, False), (9000, 9, 10, False), (5000, 1, 20, False),
                                               (3000, 1, 4, True)])
def test_compress_in_place_hole_filling(B, T, num, den, all_prot):
    """In-place compaction by hole filling, with a retained set spanning several 4096-row plan chunks, few
    holes, a short retained set and nothing to move: the retained set matches the oracle, every slot below
    n_kept that is retained stays in place, the j-th hole receives the j-th retained slot at or above
    n_kept, and every layer's K and V rows and the step / position metadata follow that plan exactly."""
    import torch
    tr = wl.custom(900 + T, L=3, Hq=4, Hkv=2, d=64, T=T, W=16, n_steps=14, budget=wl.Budget.ratio(num, den))
    if all_prot:
        tr.prot = np.ones(tr.T, np.uint8)
    g = TL.GpuTraj(tr)
    src = ([TL.bits_of(k) for k in g.K], [TL.bits_of(v) for v in g.V])
    g.problem()
    prob = B.Problem(g.K, g.V, g.Q, tr.T, g.step_id, g.prot, g.steps(), g.budget(), g.K, g.V, g.out,
                     pos_in=g.pos, step_id_out=g.step_id_out, pos_out=g.pos_out)
    st = B.stepkv_compress([prob], B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    TL.check_select_outputs(g, TL.run_oracle(tr, TL.oracle_params(B.Params())))
    n = int(g.out.n_kept.item())
    gk = g.out.kept_idx[:n].cpu().numpy().astype(np.int64)
    in_place = np.zeros(n, bool)
    in_place[gk[gk < n]] = True
    holes = np.flatnonzero(~in_place)
    movers = gk[gk >= n]
    assert len(holes) == len(movers)
    if all_prot:
        assert n == tr.T and len(holes) == 0
    exp = np.arange(n)
    exp[holes] = movers
    assert np.array_equal(g.pos_out[:n].cpu().numpy(), tr.pos[exp])
    assert np.array_equal(g.step_id_out[:n].cpu().numpy(), tr.step_id[exp])
    for l in range(tr.shape.L):
        assert np.array_equal(TL.bits_of(g.K[l])[:, :n], src[0][l][:, exp])
        assert np.array_equal(TL.bits_of(g.V[l])[:, :n], src[1][l][:, exp])


def test_compress_in_place_overflow_moves_nothing(B):
    """In place with kept_cap below the retained count (Eq. 1's protected + budget rows): the call records
    STEPKV_ENOSPACE on the device, lays out no plan, and leaves every layer's cache rows and the step /
    position outputs as they were."""
    import torch
    tr = wl.custom(77, L=2, Hq=4, Hkv=2, d=64, T=3000, W=16, n_steps=10, budget=wl.Budget.ratio(1, 2))
    n_prot = int(tr.prot.sum())
    n_exp = n_prot + max(1, (tr.T - n_prot) // 2)
    g = TL.GpuTraj(tr, kept_cap=n_exp - 7)
    src = ([TL.bits_of(k) for k in g.K], [TL.bits_of(v) for v in g.V])
    g.problem()
    prob = B.Problem(g.K, g.V, g.Q, tr.T, g.step_id, g.prot, g.steps(), g.budget(), g.K, g.V, g.out,
                     pos_in=g.pos, step_id_out=g.step_id_out, pos_out=g.pos_out)
    st = B.stepkv_compress([prob], B.Params())
    torch.cuda.synchronize()
    assert st.item() == B.STEPKV_ENOSPACE
    assert int(g.out.n_kept.item()) == n_exp
    for l in range(tr.shape.L):
        assert np.array_equal(TL.bits_of(g.K[l]), src[0][l])
        assert np.array_equal(TL.bits_of(g.V[l]), src[1][l])
    assert bool((g.step_id_out == -7).all()) and bool((g.pos_out == -7).all())


def test_compress_minimal_outputs_same_selection(B):
    """Without the optional outputs (per-step statistics, priorities) the kernel skips their work; the
    retained set and the compacted rows are the same as with every output requested."""
    import torch
    tr = wl.custom(404, L=3, Hq=8, Hkv=2, d=128, T=9000, W=32, n_steps=12, budget=wl.Budget.ratio(1, 8))
    g = TL.GpuTraj(tr)
    full = g.problem()
    st = B.stepkv_compress([full], B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    n = int(g.out.n_kept.item())
    kept_full = g.out.kept_idx[:n].clone()
    K0 = [k[:, :n].clone() for k in g.K_out]
    lean = g.problem()
    g.out = B.SelectOutputs.allocate(tr.T, tr.n_steps, g.kept_cap, "cuda", full=False)
    lean.out = g.out
    lean.refresh()
    st = B.stepkv_compress([lean], B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    assert int(g.out.n_kept.item()) == n
    assert torch.equal(g.out.kept_idx[:n], kept_full)
    for l in range(tr.shape.L):
        assert torch.equal(g.K_out[l][:, :n], K0[l])


def test_compress_all_protected(B):
    """N_t = 0: nothing is prunable, every slot is kept, B_t = 0."""
    import torch
    tr = wl.custom(3, L=2, Hq=4, Hkv=2, d=64, T=500, W=16, n_steps=2)
    tr.prot = np.ones(tr.T, np.uint8)
    g, out, _ = _compress_and_check(B, tr)
    assert out["N"] == 0 and out["B"] == 0 and int(g.out.n_kept.item()) == tr.T


def test_compress_step_without_prunable_tokens(B):
    tr = wl.custom(8, L=2, Hq=4, Hkv=2, d=64, T=2500, W=16, n_steps=6)
    k = 2
    tr.prot = tr.prot.copy()
    tr.prot[tr.step_id == k] = 1
    g, out, _ = _compress_and_check(B, tr)
    assert out["step_count"][k] == 0 and g.out.step_count[k].item() == 0


def test_compress_single_step(B):
    tr = wl.custom(12, L=1, Hq=4, Hkv=1, d=128, T=900, W=32, n_steps=1, budget=wl.Budget.ratio(1, 3))
    _compress_and_check(B, tr)


def test_compress_kept_cap_too_small(B):
    import torch
    tr = wl.tiny(1)
    g = TL.GpuTraj(tr, kept_cap=100)
    st = B.stepkv_compress([g.problem()], B.Params())
    torch.cuda.synchronize()
    assert st.item() == B.STEPKV_ENOSPACE


def test_compress_deterministic(B):
    import torch
    tr = wl.custom(31, L=3, Hq=8, Hkv=2, d=128, T=5000, W=64, n_steps=10)
    res = []
    for _ in range(2):
        g = TL.GpuTraj(tr)
        B.stepkv_compress([g.problem()], B.Params())
        torch.cuda.synchronize()
        n = int(g.out.n_kept.item())
        res.append([g.out.kept_idx[:n].cpu(), g.out.priority.cpu(), g.out.token_sal.cpu(), g.out.step_sal_sum.cpu(),
                    g.K_out[0][:, :n].cpu(), g.V_out[2][:, :n].cpu()])
    for a, b in zip(*res):
        assert torch.equal(a.contiguous().view(torch.uint8), b.contiguous().view(torch.uint8))


@pytest.mark.slow
def test_compress_full_32k_32layer(B):
    """The benchmark's workload (Llama-3-8B shape, T = 32768, 32 layers, 10% budget), in the same
    fused call the benchmark times: saliency layers from the shared generator, the other layers'
    K/V drawn on the device; selection checked against the oracle, compaction checked row for row
    against the oracle's retained slots."""
    import torch
    tr = wl.llama8b_32k(seed=1)
    s = tr.shape
    gen = torch.Generator(device="cuda").manual_seed(1234)
    sal_ids = set(tr.sal_layer_ids())
    K = [TL.bf16_dev(tr.keys(l)) if l in sal_ids else
         torch.randn((s.Hkv, s.T, s.d), generator=gen, device="cuda", dtype=torch.bfloat16) for l in range(s.L)]
    V = [torch.randn((s.Hkv, s.T, s.d), generator=gen, device="cuda", dtype=torch.bfloat16) for _ in range(s.L)]
    g = TL.GpuTraj.__new__(TL.GpuTraj)
    g.tr = tr
    g.K, g.V = K, V
    g.Q = [TL.bf16_dev(tr.queries(l)) for l in tr.sal_layer_ids()]
    for nm, arr in (("step_id", tr.step_id), ("prot", tr.prot), ("pos", tr.pos), ("valid", tr.valid),
                    ("gain", tr.gain), ("red", tr.red), ("obs_sim", tr.obs_sim), ("reuse_in", tr.reuse)):
        setattr(g, nm, torch.from_numpy(arr).cuda())
    g.reuse_out = torch.empty_like(g.reuse_in)
    g.kept_cap = 4096
    prob = g.problem()
    st = B.stepkv_compress([prob], B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    out = TL.run_oracle(tr, TL.oracle_params(B.Params()))
    swaps = TL.check_select_outputs(g, out)
    n = int(g.out.n_kept.item())
    assert n == 16 + 64 + 3268
    kept = g.out.kept_idx[:n].long()
    for l in range(s.L):
        assert torch.equal(g.K_out[l][:, :n], K[l].index_select(1, kept))
        assert torch.equal(g.V_out[l][:, :n], V[l].index_select(1, kept))
    print(f"full-size swaps: {swaps}")


def test_compress_batched_short_trajectories(B):
    """Short trajectories of one head shape share one saliency launch (lengths and strides differ; a
    different shape in the middle starts a new launch); every trajectory matches the oracle."""
    import torch
    shapes = [(64, 1200), (64, 2048), (64, 777), (128, 1500), (64, 3100), (64, 2500), (64, 1000), (64, 640),
              (64, 1800), (64, 2222)]
    trs = [wl.custom(200 + i, L=2, Hq=8, Hkv=2, d=d, T=T, W=24, n_steps=4 + i % 5, budget=wl.Budget.ratio(1, 4))
           for i, (d, T) in enumerate(shapes)]
    gs = [TL.GpuTraj(tr) for tr in trs]
    probs = [g.problem() for g in gs]
    st = B.stepkv_compress(probs, B.Params())
    torch.cuda.synchronize()
    assert st.item() == 0
    for g, tr in zip(gs, trs):
        out = TL.run_oracle(tr, TL.oracle_params(B.Params()))
        TL.check_select_outputs(g, out)
        n = int(g.out.n_kept.item())
        gk = g.out.kept_idx[:n].cpu().numpy()
        for l in range(tr.shape.L):
            assert np.array_equal(TL.bits_of(g.K_out[l])[:, :n], O.compact_rows(tr.keys(l), gk))
            assert np.array_equal(TL.bits_of(g.V_out[l])[:, :n], O.compact_rows(tr.values(l), gk))


def test_compress_stage_events(B):
    """stepkv_set_stage_events: a pass records the caller's three events around its stages and its
    results equal those of a pass without them; clearing the events stops the recording."""
    import torch
    tr = wl.custom(95, L=4, Hq=16, Hkv=4, d=128, T=6000, W=64, n_steps=10, budget=wl.Budget.ratio(1, 10))
    g1, g2 = TL.GpuTraj(tr), TL.GpuTraj(tr)
    p1, p2 = g1.problem(), g2.problem()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    for e in ev:
        e.record()
    torch.cuda.synchronize()
    B.set_stage_events(*ev)
    B.stepkv_compress([p1], B.Params())
    B.set_stage_events()
    after = torch.cuda.Event(enable_timing=True)
    B.stepkv_compress([p2], B.Params())
    after.record()
    torch.cuda.synchronize()
    t_sal_sel, t_compact = ev[0].elapsed_time(ev[1]), ev[1].elapsed_time(ev[2])
    assert t_sal_sel > 0 and t_compact > 0
    assert ev[2].elapsed_time(after) > 0  # the second pass recorded nothing into the events
    n = int(g1.out.n_kept.item())
    assert torch.equal(g1.out.kept_idx[:n], g2.out.kept_idx[:n])
    for l in range(tr.shape.L):
        assert torch.equal(g1.K_out[l][:, :n], g2.K_out[l][:, :n])
