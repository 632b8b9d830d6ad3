"""The incremental agent loop through the C ABI: compress at a boundary, decode over the compacted cache,
append the next step to the retained rows, compress again.  Every boundary is checked against the
oracle on the same inputs (the GPU's carried cache, step ids, positions and reuse accumulators), so the
carrying of state across boundaries is exercised without letting a tolerated swap at one boundary
change what the next boundary is compared on.
"""
import types

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


@pytest.mark.parametrize("d", [64, 128])
def test_incremental_loop_four_boundaries(B, d):
    import torch
    L, Hq, Hkv, W, t0, budget = 3, 8, 2, 16, 1200, 300
    lp = wl.IncrementalLoop(7 + d, L=L, Hq=Hq, Hkv=Hkv, d=d, W=W, t0=t0, budget_count=budget)
    step_id, n_steps = lp.initial_layout()
    pos = np.arange(t0, dtype=np.int32)
    next_pos = t0
    K = [lp.rows(0, l, wl._K_KEYS, t0) for l in range(L)]
    V = [lp.rows(0, l, wl._K_VALUES, t0) for l in range(L)]
    reuse = np.zeros(n_steps, np.float32)
    p = B.Params()
    sal_ids = list(range(L - min(3, L), L))
    for b in range(4):
        if b > 0:
            n_new = lp.step_length(b)
            n_steps += 1
            K = [np.concatenate([k, lp.rows(b, l, wl._K_KEYS, n_new)], axis=1) for l, k in enumerate(K)]
            V = [np.concatenate([v, lp.rows(b, l, wl._K_VALUES, n_new)], axis=1) for l, v in enumerate(V)]
            step_id = np.concatenate([step_id, np.full(n_new, n_steps - 1, np.int32)])
            pos = np.concatenate([pos, np.arange(next_pos, next_pos + n_new, dtype=np.int32)])
            next_pos += n_new
            reuse = np.concatenate([reuse, np.float32([0.5])])  # stale: Algorithm 1 resets c_t
        T = step_id.shape[0]
        prot = lp.protected(step_id)
        valid, gain, red, obs_sim = lp.signals(b, n_steps)
        Q = [lp.queries(b, l) for l in sal_ids]
        dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
        Kd = [TL.bf16_dev(k) for k in K]
        Vd = [TL.bf16_dev(v) for v in V]
        reuse_out = torch.empty(n_steps, dtype=torch.float32, device="cuda")
        steps = B.StepSignals(dev(valid), dev(gain), dev(red), dev(reuse), dev(obs_sim), reuse_out)
        cap = T
        out = B.SelectOutputs.allocate(T, n_steps, cap, "cuda")
        K_out = [torch.empty((Hkv, cap, d), dtype=torch.bfloat16, device="cuda") for _ in range(L)]
        V_out = [torch.empty((Hkv, cap, d), dtype=torch.bfloat16, device="cuda") for _ in range(L)]
        sid_out = torch.empty(cap, dtype=torch.int32, device="cuda")
        pos_out = torch.empty(cap, dtype=torch.int32, device="cuda")
        prob = B.Problem(Kd, Vd, [TL.bf16_dev(q) for q in Q], T, dev(step_id), dev(prot), steps,
                         B.budget_count(budget), K_out, V_out, out, pos_in=dev(pos), step_id_out=sid_out,
                         pos_out=pos_out)
        st = B.stepkv_compress([prob], p)
        # decode over the compacted cache right away, n read on the device
        qdec = [wl.decode_queries(100 + b, L, Hq, d, 1)[0, l] for l in range(L)]
        dec = B.stepkv_decode([TL.bf16_dev(q) for q in qdec], K_out, V_out, out.n_kept, status=st)
        torch.cuda.synchronize()
        assert st.item() == 0, b
        ref = O.compress([K[l] for l in sal_ids], Q, step_id, prot, valid, gain, red, obs_sim, reuse,
                         TL.oracle_params(p), "count", count=budget)
        g = types.SimpleNamespace(out=out, tr=types.SimpleNamespace(prot=prot), reuse_out=reuse_out)
        TL.check_select_outputs(g, ref)
        n = int(out.n_kept.item())
        assert n == int(prot.sum()) + min(budget, T - int(prot.sum()))
        kept = out.kept_idx[:n].cpu().numpy().astype(np.int64)
        kt = torch.from_numpy(kept).cuda()
        for l in range(L):
            assert torch.equal(K_out[l][:, :n], Kd[l].index_select(1, kt))
            assert torch.equal(V_out[l][:, :n], Vd[l].index_select(1, kt))
            TL.assert_decode_close(dec[l].cpu().numpy(), qdec[l], K[l][:, kept], V[l][:, kept], f"decode {b}/{l}")
        assert np.array_equal(sid_out[:n].cpu().numpy(), step_id[kept])
        assert np.array_equal(pos_out[:n].cpu().numpy(), pos[kept])
        # carry the compacted state to the next boundary
        K = [k[:, kept] for k in K]
        V = [v[:, kept] for v in V]
        step_id = step_id[kept]
        pos = pos[kept]
        reuse = reuse_out.cpu().numpy()


def test_incremental_loop_in_place(B):
    """The same loop with the cache compacted in place (hole filling) inside one capacity buffer per
    layer: each boundary's rows are checked as a set against the oracle's retained rows, through the
    original positions the pass reports, and the next step is appended after the retained rows."""
    import torch
    L, Hq, Hkv, d, W, t0, budget = 3, 8, 2, 64, 16, 1200, 300
    lp = wl.IncrementalLoop(11, L=L, Hq=Hq, Hkv=Hkv, d=d, W=W, t0=t0, budget_count=budget)
    n_b = 4
    cap_total = t0 + sum(lp.step_length(b) for b in range(1, n_b))
    Kbuf = [torch.zeros((Hkv, cap_total, d), dtype=torch.bfloat16, device="cuda") for _ in range(L)]
    Vbuf = [torch.zeros((Hkv, cap_total, d), dtype=torch.bfloat16, device="cuda") for _ in range(L)]
    step_id, n_steps = lp.initial_layout()
    pos = np.arange(t0, dtype=np.int32)
    next_pos = t0
    K = [lp.rows(0, l, wl._K_KEYS, t0) for l in range(L)]  # host mirror of the live rows, same order
    V = [lp.rows(0, l, wl._K_VALUES, t0) for l in range(L)]
    for l in range(L):
        Kbuf[l][:, :t0] = TL.bf16_dev(K[l])
        Vbuf[l][:, :t0] = TL.bf16_dev(V[l])
    reuse = np.zeros(n_steps, np.float32)
    p = B.Params()
    for b in range(n_b):
        if b > 0:
            n_new = lp.step_length(b)
            n_steps += 1
            T0 = step_id.shape[0]
            for l in range(L):
                kn, vn = lp.rows(b, l, wl._K_KEYS, n_new), lp.rows(b, l, wl._K_VALUES, n_new)
                Kbuf[l][:, T0:T0 + n_new] = TL.bf16_dev(kn)
                Vbuf[l][:, T0:T0 + n_new] = TL.bf16_dev(vn)
                K[l] = np.concatenate([K[l], kn], axis=1)
                V[l] = np.concatenate([V[l], vn], axis=1)
            step_id = np.concatenate([step_id, np.full(n_new, n_steps - 1, np.int32)])
            pos = np.concatenate([pos, np.arange(next_pos, next_pos + n_new, dtype=np.int32)])
            next_pos += n_new
            reuse = np.concatenate([reuse, np.float32([0.5])])
        T = step_id.shape[0]
        prot = lp.protected(step_id)
        valid, gain, red, obs_sim = lp.signals(b, n_steps)
        Q = [lp.queries(b, l) for l in range(L)]
        dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
        live_K = [k[:, :T] for k in Kbuf]
        live_V = [v[:, :T] for v in Vbuf]
        reuse_out = torch.empty(n_steps, dtype=torch.float32, device="cuda")
        steps = B.StepSignals(dev(valid), dev(gain), dev(red), dev(reuse), dev(obs_sim), reuse_out)
        out = B.SelectOutputs.allocate(T, n_steps, T, "cuda")
        sid_out = torch.empty(T, dtype=torch.int32, device="cuda")
        pos_out = torch.empty(T, dtype=torch.int32, device="cuda")
        prob = B.Problem(live_K, live_V, [TL.bf16_dev(q) for q in Q], T, dev(step_id), dev(prot), steps,
                         B.budget_count(budget), live_K, live_V, out, pos_in=dev(pos), step_id_out=sid_out,
                         pos_out=pos_out)
        st = B.stepkv_compress([prob], p)
        torch.cuda.synchronize()
        assert st.item() == 0, b
        ref = O.compress(K, Q, step_id, prot, valid, gain, red, obs_sim, reuse, TL.oracle_params(p), "count",
                         count=budget)
        g = types.SimpleNamespace(out=out, tr=types.SimpleNamespace(prot=prot), reuse_out=reuse_out)
        TL.check_select_outputs(g, ref)
        n = int(out.n_kept.item())
        kept = out.kept_idx[:n].cpu().numpy().astype(np.int64)
        # rows [0, n) hold the retained set: slot r came from slot src[r] (r itself when retained below n)
        pos_of_slot = {int(pp): i for i, pp in enumerate(pos)}
        po = pos_out[:n].cpu().numpy()
        src = np.array([pos_of_slot[int(x)] for x in po])
        assert np.array_equal(np.sort(src), kept)
        below = kept[kept < n]
        assert np.array_equal(src[below], below)  # retained rows below n did not move
        assert np.array_equal(sid_out[:n].cpu().numpy(), step_id[src])
        for l in range(L):
            assert np.array_equal(TL.bits_of(Kbuf[l][:, :n]), K[l][:, src])
            assert np.array_equal(TL.bits_of(Vbuf[l][:, :n]), V[l][:, src])
        K = [k[:, src] for k in K]
        V = [v[:, src] for v in V]
        step_id = step_id[src]
        pos = pos[src]
        reuse = reuse_out.cpu().numpy()


@pytest.mark.slow
def test_incremental_loop_llama_heads_two_oracle_chains(B):
    """Ten boundaries at Llama-3-8B head shapes (Hq 32, Hkv 8, d 128, W 64) under the 8192-token budget,
    the cache compacted in place and decoded after every compression.

    Chain A checks each boundary against the oracle run on the state the GPU carried (its retained rows,
    step ids, positions and fp32 reuse accumulators), so one boundary's result is never judged on
    another's.  Chain B is the oracle alone, carrying its own retained set and fp64 accumulators from
    the first boundary on; the GPU's retained positions must equal chain B's at every boundary and its
    accumulators stay within the parity tolerance of chain B's, so drift over the loop would show."""
    import torch
    L, Hq, Hkv, d, W, budget = 3, 32, 8, 128, 64, 8192
    t0 = budget + 16 + W + 700
    n_b = 10
    lp = wl.IncrementalLoop(23, L=L, Hq=Hq, Hkv=Hkv, d=d, W=W, t0=t0, budget_count=budget)
    cap = t0 + max(lp.step_length(b) for b in range(1, n_b)) + 16
    Kbuf = [torch.zeros((Hkv, cap, d), dtype=torch.bfloat16, device="cuda") for _ in range(L)]
    Vbuf = [torch.zeros((Hkv, cap, d), dtype=torch.bfloat16, device="cuda") for _ in range(L)]
    step_id, n_steps = lp.initial_layout()
    pos = np.arange(t0, dtype=np.int32)
    next_pos = t0
    K = [lp.rows(0, l, wl._K_KEYS, t0) for l in range(L)]  # chain A: host mirror of the GPU's live rows
    V = [lp.rows(0, l, wl._K_VALUES, t0) for l in range(L)]
    for l in range(L):
        Kbuf[l][:, :t0] = TL.bf16_dev(K[l])
        Vbuf[l][:, :t0] = TL.bf16_dev(V[l])
    reuse = np.zeros(n_steps, np.float32)
    # chain B: positions, step ids and accumulators of the oracle-only trajectory (rows looked up by position)
    pos_b, sid_b, reuse_b = pos.copy(), step_id.copy(), np.zeros(n_steps)
    p = B.Params()
    po_ = TL.oracle_params(p)
    dev = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    st = B.new_status()
    ws = None
    for b in range(n_b):
        if b > 0:
            n_new = lp.step_length(b)
            n_steps += 1
            T0 = step_id.shape[0]
            new_pos = np.arange(next_pos, next_pos + n_new, dtype=np.int32)
            for l in range(L):
                kn, vn = lp.rows(b, l, wl._K_KEYS, n_new), lp.rows(b, l, wl._K_VALUES, n_new)
                Kbuf[l][:, T0:T0 + n_new] = TL.bf16_dev(kn)
                Vbuf[l][:, T0:T0 + n_new] = TL.bf16_dev(vn)
                K[l] = np.concatenate([K[l], kn], axis=1)
                V[l] = np.concatenate([V[l], vn], axis=1)
            step_id = np.concatenate([step_id, np.full(n_new, n_steps - 1, np.int32)])
            pos = np.concatenate([pos, new_pos])
            pos_b = np.concatenate([pos_b, new_pos])
            sid_b = np.concatenate([sid_b, np.full(n_new, n_steps - 1, np.int32)])
            next_pos += n_new
            reuse = np.concatenate([reuse, np.float32([0.5])])
            reuse_b = np.concatenate([reuse_b, [0.5]])
        T = step_id.shape[0]
        prot = lp.protected(step_id)
        valid, gain, red, obs_sim = lp.signals(b, n_steps)
        Q = [lp.queries(b, l) for l in range(L)]
        live_K = [k[:, :T] for k in Kbuf]
        live_V = [v[:, :T] for v in Vbuf]
        reuse_out = torch.empty(n_steps, dtype=torch.float32, device="cuda")
        steps = B.StepSignals(dev(valid), dev(gain), dev(red), dev(reuse), dev(obs_sim), reuse_out)
        kcap = min(T, budget + int(prot.sum()))
        out = B.SelectOutputs.allocate(T, n_steps, kcap, "cuda")
        sid_out = torch.empty(kcap, dtype=torch.int32, device="cuda")
        pos_out = torch.empty(kcap, dtype=torch.int32, device="cuda")
        prob = B.Problem(live_K, live_V, [TL.bf16_dev(q) for q in Q], T, dev(step_id), dev(prot), steps,
                         B.budget_count(budget), live_K, live_V, out, pos_in=dev(pos), step_id_out=sid_out,
                         pos_out=pos_out)
        need = B.stepkv_workspace_size([prob])
        if ws is None or ws.numel() < need:
            ws = torch.empty(need + (1 << 20), dtype=torch.uint8, device="cuda")
        B.stepkv_compress([prob], p, ws=ws, status=st)
        qdec = [wl.decode_queries(300 + b, L, Hq, d, 1)[0, l] for l in range(L)]
        dec = B.stepkv_decode([TL.bf16_dev(q) for q in qdec], live_K, live_V, out.n_kept, status=st)
        torch.cuda.synchronize()
        assert st.item() == 0, b
        # chain A: the oracle on the GPU-carried state
        ref = O.compress(K, Q, step_id, prot, valid, gain, red, obs_sim, reuse, po_, "count", count=budget)
        g = types.SimpleNamespace(out=out, tr=types.SimpleNamespace(prot=prot), reuse_out=reuse_out)
        swaps = TL.check_select_outputs(g, ref)
        n = int(out.n_kept.item())
        kept = out.kept_idx[:n].cpu().numpy().astype(np.int64)
        slot_of_pos = {int(pp): i for i, pp in enumerate(pos)}
        src = np.array([slot_of_pos[int(x)] for x in pos_out[:n].cpu().numpy()])
        assert np.array_equal(np.sort(src), kept)
        assert np.array_equal(sid_out[:n].cpu().numpy(), step_id[src])
        for l in range(L):
            assert np.array_equal(TL.bits_of(Kbuf[l][:, :n]), K[l][:, src])
            assert np.array_equal(TL.bits_of(Vbuf[l][:, :n]), V[l][:, src])
            TL.assert_decode_close(dec[l].cpu().numpy(), qdec[l], K[l][:, src], V[l][:, src], f"decode {b}/{l}")
        # chain B: the oracle-only trajectory.  While its rows are the same set as chain A's, its saliency
        # per key is chain A's (the window rows are the last W of both, and every other key is visible to
        # every window query, so a key's saliency does not depend on the order of the rows).
        assert np.array_equal(np.sort(pos_b), np.sort(pos)), f"chains diverged before boundary {b}"
        perm = np.array([slot_of_pos[int(x)] for x in pos_b])  # chain-B slot -> chain-A slot
        prot_b = lp.protected(sid_b)
        assert np.array_equal(prot_b, prot[perm])
        ref_b = O.stepkv_boundary([a[:, perm] for a in ref["A"]], sid_b, prot_b, valid, gain, red, obs_sim, reuse_b,
                                  po_, "count", count=budget)
        gpu_pos = np.sort(pos[kept])
        if swaps == 0:
            assert np.array_equal(gpu_pos, np.sort(pos_b[ref_b["kept"]])), f"retained set drifted at boundary {b}"
        TL.assert_close(reuse_out.cpu().numpy(), ref_b["reuse"], f"c_k vs oracle-only chain at boundary {b}",
                        floor=1e-6)
        TL.assert_close(out.step_util.cpu().numpy(), ref_b["S"], f"S_k vs oracle-only chain at boundary {b}",
                        floor=1e-6)
        # carry both chains to the next boundary
        K = [k[:, src] for k in K]
        V = [v[:, src] for v in V]
        step_id = step_id[src]
        pos = pos[src]
        reuse = reuse_out.cpu().numpy()
        kb = ref_b["kept"]
        pos_b, sid_b, reuse_b = pos_b[kb], sid_b[kb], ref_b["reuse"]
