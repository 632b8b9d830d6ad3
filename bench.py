"""Benchmark of the fused StepKV compression pass (score -> reduce/fuse -> select -> compact).

Workload (default): one Llama-3-8B-shaped trajectory per GPU -- 32 layers, 32 query / 8 KV heads,
head dim 128, bf16, T = 32768 cached tokens, 40 reasoning steps, 64-token observation window,
budget 10% of the prunable tokens -- drawn by the seeded generator (saliency layers, step layout,
signals) and by torch's seeded device RNG (K/V of the other layers).  Inputs are resident in HBM when
the timed region starts; an L2 flush (a 512 MB write) runs between timed steps, outside their events.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line (rank 0).  Under torchrun (N > 1) every rank compresses its own trajectory
(independent problems: weak scaling, no collective on the data path); timing is the max over ranks.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "compressed tokens/sec (score+select+compact) at 32K ctx; % HBM roofline"
UNIT = "tokens/s"


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


# ---------------------------------------------------------------------------------- workload
def make_traj(args):
    from paper_2609_22158_gb300 import workload as wl
    return wl.llama8b_32k(seed=args.seed, T=args.T, L=args.layers)


def workload_config(tr, args, n):
    s = tr.shape
    b = tr.budget
    return {
        "workload": (f"llama3-8b-shaped agent trajectory: L={s.L}, Hq={s.Hq}, Hkv={s.Hkv}, d={s.d}, T={s.T}, "
                     f"W={s.W}, {tr.n_steps} steps, saliency from last {s.Ls} layers, budget "
                     + (f"{b.num}/{b.den} of prunable" if b.mode == "ratio" else f"{b.count} tokens")),
        "global_batch": n, "seq_len": s.T, "parallelism": f"dp{n} (independent trajectories)",
        "l2": "flushed between timed steps (512 MB write outside the step events); inputs 4 GB > L2",
    }


class DeviceTraj:
    """Device-resident inputs/outputs of one trajectory and the C-ABI problem descriptor."""

    def __init__(self, tr, device, seed=1234):
        import numpy as np
        import torch
        from paper_2609_22158_gb300 import binding as B
        self.tr = tr
        s = tr.shape
        gen = torch.Generator(device=device).manual_seed(seed)
        sal_ids = set(tr.sal_layer_ids())

        def bf16(bits):
            return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(device)

        self.K = [bf16(tr.keys(l)) if l in sal_ids else
                  torch.randn((s.Hkv, s.T, s.d), generator=gen, device=device, dtype=torch.bfloat16)
                  for l in range(s.L)]
        self.V = [torch.randn((s.Hkv, s.T, s.d), generator=gen, device=device, dtype=torch.bfloat16)
                  for _ in range(s.L)]
        self.Q = [bf16(tr.queries(l)) for l in tr.sal_layer_ids()]
        t = lambda a: torch.from_numpy(a).to(device)
        self.step_id, self.prot, self.pos = t(tr.step_id), t(tr.prot), t(tr.pos)
        self.steps = B.StepSignals(t(tr.valid), t(tr.gain), t(tr.red), t(tr.reuse), t(tr.obs_sim),
                                   torch.empty(tr.n_steps, dtype=torch.float32, device=device))
        n_prot = int(tr.prot.sum())
        N = s.T - n_prot
        B_t = (max(1, tr.budget.num * N // tr.budget.den) if tr.budget.mode == "ratio" else tr.budget.count)
        self.n_kept_expected = n_prot + min(B_t, N)
        self.cap = self.n_kept_expected
        self.K_out = [torch.empty((s.Hkv, self.cap, s.d), dtype=torch.bfloat16, device=device) for _ in range(s.L)]
        self.V_out = [torch.empty((s.Hkv, self.cap, s.d), dtype=torch.bfloat16, device=device) for _ in range(s.L)]
        self.out = B.SelectOutputs.allocate(s.T, tr.n_steps, self.cap, device, full=False)
        self.step_id_out = torch.empty(self.cap, dtype=torch.int32, device=device)
        self.pos_out = torch.empty(self.cap, dtype=torch.int32, device=device)
        b = tr.budget
        self.budget = B.budget_ratio(b.num, b.den) if b.mode == "ratio" else B.budget_count(b.count)
        self.problem = B.Problem(self.K, self.V, self.Q, s.T, self.step_id, self.prot, self.steps, self.budget,
                                 self.K_out, self.V_out, self.out, pos_in=self.pos, step_id_out=self.step_id_out,
                                 pos_out=self.pos_out)
        self.ws = torch.empty(B.stepkv_workspace_size([self.problem]) + 512, dtype=torch.uint8, device=device)
        self.status = B.new_status(device)

    def compress(self, params, stream=None):
        from paper_2609_22158_gb300 import binding as B
        B.stepkv_compress([self.problem], params, ws=self.ws, status=self.status, stream=stream)


def launches_per_pass(tr) -> int:
    """Kernel launches of one stepkv_compress call (mirrors the library's launch plan)."""
    s = tr.shape
    return 1 + 1 + math.ceil(s.L / 96)  # score (both passes, one cooperative launch), select, compaction


def algorithmic_bytes(tr, n_kept):
    """Bytes the pass must move at minimum (stage by stage)."""
    s = tr.shape
    G = s.Hq // s.Hkv
    score = s.Ls * s.Hkv * s.T * s.d * 2 + s.Ls * s.Hq * s.W * s.d * 2 + s.Ls * s.Hkv * s.T * 4
    select = s.Ls * s.Hkv * s.T * 4 + s.T * (4 + 1) + n_kept * 4
    compact = 2 * s.L * s.Hkv * n_kept * s.d * 2 * 2 + n_kept * 4 * 3
    return {"score": score, "select": select, "compact": compact, "total": score + select + compact}


# ---------------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.path = tempfile.mktemp(suffix=".csv")
        self.proc = None
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "100", "-i", str(gpu_index)], stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        self.marks = []

    def mark(self, name):
        self.marks.append((name, time.time()))

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    try:
                        rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
                    except ValueError:
                        pass
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        loaded = [r for r in rows if r[0] > 0.5 * r[1]] or rows
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i, v in enumerate(r[2]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in loaded), "sm_max_mhz": max(r[1] for r in rows),
                "samples": len(rows), "reasons": reasons}


# ---------------------------------------------------------------------------------- oracle timing
ORACLE_SNIPPET = r"""
import json, sys, time
sys.path.insert(0, {root!r})
import numpy as np
from oracle import stepkv_oracle as O
from paper_2609_22158_gb300 import workload as wl
tr = wl.llama8b_32k(seed={seed}, T={T}, L={L})
s = tr.shape
pairs = {pairs}
Ks = [tr.keys(l) for l in tr.sal_layer_ids()]
Qs = [tr.queries(l) for l in tr.sal_layer_ids()]
V0 = tr.values(tr.sal_layer_ids()[0])
G = s.Hq // s.Hkv
t0 = time.perf_counter()
A = []
done = 0
for li in range(len(Ks)):
    rows = []
    for h in range(s.Hkv):
        if done < pairs:
            rows.append(O.window_attention_saliency(Ks[li][h:h + 1], Qs[li][h * G:(h + 1) * G])[0])
            done += 1
        else:
            rows.append(np.zeros(s.T))
    A.append(np.stack(rows))
t1 = time.perf_counter()
b = tr.budget
out = O.stepkv_boundary(A, tr.step_id, tr.prot, tr.valid, tr.gain, tr.red, tr.obs_sim, tr.reuse, O.Params(),
                        b.mode, b.num, b.den, b.count)
t2 = time.perf_counter()
for rep in range({compact_sets}):
    C = O.compact_rows(V0[rep % s.Hkv:rep % s.Hkv + 1], out["kept"])
t3 = time.perf_counter()
print(json.dumps({{"score_s": t1 - t0, "select_s": t2 - t1, "compact_s": t3 - t2, "n_kept": int(len(out["kept"]))}}))
"""


def oracle_pass_seconds(args, pairs: int, compact_sets: int, threads: int = 1):
    """Run the oracle (as it stands) on a bounded sample in a fresh single-threaded process and scale
    each stage to the whole pass.  Returns (seconds per full pass, description, threads)."""
    from paper_2609_22158_gb300 import workload as wl
    tr = make_traj(args)
    s = tr.shape
    code = ORACLE_SNIPPET.format(root=ROOT, seed=args.seed, T=args.T, L=args.layers, pairs=pairs,
                                 compact_sets=compact_sets)
    env = dict(os.environ)
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "NUMEXPR_NUM_THREADS"):
        env[k] = str(threads)
    env["CUDA_VISIBLE_DEVICES"] = ""
    r = subprocess.run([sys.executable, "-c", code], stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True,
                       env=env, timeout=1800)
    if r.returncode != 0:
        raise RuntimeError("oracle run failed: " + r.stderr[-2000:])
    m = json.loads(r.stdout.strip().splitlines()[-1])
    n_pairs = s.Ls * s.Hkv
    n_sets = 2 * s.L * s.Hkv
    total = m["score_s"] * n_pairs / pairs + m["select_s"] + m["compact_s"] * n_sets / compact_sets
    desc = (f"oracle (numpy fp64, {threads} thread) on the same workload: saliency of {pairs} of {n_pairs} "
            f"(layer, KV head) pairs, full selection, compaction of {compact_sets} of {n_sets} (layer, tensor, head) "
            f"row sets; each stage's time scaled to the whole pass")
    return total, desc, m


# ---------------------------------------------------------------------------------- ours
def run_ours(args):
    import numpy as np
    import torch
    from paper_2609_22158_gb300 import binding as B

    from paper_2609_22158_gb300 import multirank as MR
    world, rank, local = MR.rank_env()
    dist = None
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(dev)
    from paper_2609_22158_gb300 import build
    build.build_library()
    B.load_library()

    tr = make_traj(args)
    s = tr.shape
    dt = DeviceTraj(tr, dev, seed=MR.rank_seed(1234, rank))
    params = B.Params()
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(512 * 1024 * 1024, dtype=torch.uint8, device=dev)
    hbm, _, peak_kind = _peaks()

    sampler = ClockSampler(dev.index if world == 1 else local) if rank == 0 else None

    # warm-up
    for _ in range(args.warmup):
        dt.compress(params, stream)
        flush.fill_(1)
    torch.cuda.synchronize()
    st = int(dt.status.item())
    if st != 0:
        raise RuntimeError(f"device status {st} after warm-up")
    n_kept = int(dt.out.n_kept.item())
    assert n_kept == dt.n_kept_expected, (n_kept, dt.n_kept_expected)

    # timed region: exactly K fused passes, each bracketed by CUDA events on the launching stream
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    if sampler:
        sampler.mark("timed_start")
    wall0 = time.perf_counter()
    for i in range(args.steps):
        ev[i][0].record(stream)
        dt.compress(params, stream)
        ev[i][1].record(stream)
        flush.fill_(i & 0xFF)
    torch.cuda.synchronize()
    wall1 = time.perf_counter()
    if dist:
        dist.barrier()
    step_ms = [a.elapsed_time(b) for a, b in ev]
    ms = MR.max_over_ranks(sum(step_ms) / len(step_ms), dist, dev)
    if int(dt.status.item()) != 0:
        raise RuntimeError(f"device status {int(dt.status.item())} in the timed region")
    tokens = MR.gather_tokens(s.T, dist, dev)
    value = MR.job_throughput(tokens, ms * 1e-3)

    # per-stage timing (same shapes, separate entry points, same stream) for the roofline
    stage = {}
    if rank == 0 and not args.no_stages:
        sal = torch.empty((s.Ls, s.Hkv, s.T), dtype=torch.float32, device=dev)
        ws_s = torch.empty(B.load_library().stepkv_score_workspace_size(s.Ls, s.Hkv, s.Hq, s.T, s.W) + 512,
                           dtype=torch.uint8, device=dev)
        ws_sel = torch.empty(B.load_library().stepkv_select_workspace_size(s.Ls * s.Hkv, s.T, tr.n_steps) + 512,
                             dtype=torch.uint8, device=dev)
        sel_out = B.SelectOutputs.allocate(s.T, tr.n_steps, dt.cap, dev, full=False)
        Ksal = [dt.K[l] for l in tr.sal_layer_ids()]
        reps = max(3, min(args.steps, 20))
        times = {"score": [], "select": [], "compact": []}
        for r in range(reps + 2):
            e = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
            flush.fill_(r & 0xFF)
            torch.cuda._sleep(200_000)
            e[0].record(stream)
            B.stepkv_score(Ksal, dt.Q, s.T, sal=sal, ws=ws_s, status=dt.status, stream=stream)
            e[1].record(stream)
            B.stepkv_select(sal, dt.step_id, dt.prot, dt.steps, params, dt.budget, sel_out, ws=ws_sel,
                            status=dt.status, stream=stream)
            e[2].record(stream)
            flush.fill_((r + 1) & 0xFF)
            # keep the device busy while the host marshals the 64 per-layer tensors of the call, so the
            # events time the kernel and not the host
            torch.cuda._sleep(400_000)
            e3 = torch.cuda.Event(enable_timing=True)
            e3.record(stream)
            B.stepkv_compact(dt.K, dt.V, s.T, sel_out.kept_idx, sel_out.n_kept, dt.cap, dt.K_out, dt.V_out,
                             dt.step_id, dt.pos, dt.step_id_out, dt.pos_out, status=dt.status, stream=stream)
            e[3].record(stream)
            torch.cuda.synchronize()
            if r >= 2:
                times["score"].append(e[0].elapsed_time(e[1]))
                times["select"].append(e[1].elapsed_time(e[2]))
                times["compact"].append(e3.elapsed_time(e[3]))
        stage = {k: statistics.median(v) * 1e3 for k, v in times.items()}  # us

    # e2e: host buffers through the same public call.  The cache lives in page-locked host memory and the
    # compacted cache is written back to host memory: every step copies the window queries, the token
    # metadata and the saliency layers' K host->device, the compaction reads the retained rows of all
    # layers across the CPU-GPU link and writes them to the host outputs, and the retained slots come back
    # device->host.  The second figure copies every input to the device and every output back instead.
    e2e = None
    e2e_copy_all = None
    if not args.no_e2e:
        s_ = tr.shape
        host_K = [t.cpu().pin_memory() for t in dt.K]
        host_V = [t.cpu().pin_memory() for t in dt.V]
        host_Q = [t.cpu().pin_memory() for t in dt.Q]
        host_small = [x.cpu().pin_memory() for x in (dt.step_id, dt.prot, dt.pos)]
        dev_small = [dt.step_id, dt.prot, dt.pos]
        sal_ids = list(tr.sal_layer_ids())
        K_sal = [torch.empty_like(dt.K[l]) for l in sal_ids]
        host_Kout = [torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in dt.K_out]
        host_Vout = [torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in dt.V_out]
        host_idx = torch.empty(dt.cap + 1, dtype=torch.int32).pin_memory()
        sig_dev = [dt.steps.valid, dt.steps.gain, dt.steps.red, dt.steps.reuse_in, dt.steps.obs_sim]
        host_sig = [x.cpu().pin_memory() for x in sig_dev]
        nb = lambda ts: sum(t.numel() * t.element_size() for t in ts)
        row_bytes = 2 * s_.L * s_.Hkv * s_.d * 2  # K and V of one retained slot, all layers
        k2 = max(1, min(args.steps, args.e2e_steps))
        # Two sets of device input buffers, so that the next step's host->device copies (on their own
        # stream) run while the current step gathers its rows across the link in the other direction.
        copy_stream = torch.cuda.Stream(device=dev)
        bufs = []
        for _ in range(2):
            Qb = [torch.empty_like(q) for q in dt.Q]
            smallb = [torch.empty_like(x) for x in dev_small]
            sigb = [torch.empty_like(x) for x in sig_dev]
            Ksb = [torch.empty_like(dt.K[l]) for l in sal_ids]
            stepsb = B.StepSignals(sigb[0], sigb[1], sigb[2], sigb[3], sigb[4], dt.steps.reuse_out)
            probb = B.Problem(host_K, host_V, Qb, s_.T, smallb[0], smallb[1], stepsb, dt.budget, host_Kout,
                              host_Vout, dt.out, pos_in=smallb[2], step_id_out=dt.step_id_out, pos_out=dt.pos_out,
                              kv_location=B.STEPKV_MEM_HOST, out_location=B.STEPKV_MEM_HOST, K_sal=Ksb)
            bufs.append((Qb + smallb + sigb + Ksb, probb, torch.cuda.Event(), torch.cuda.Event()))
        step_inputs = host_Q + host_small + host_sig + [host_K[l] for l in sal_ids]
        n_step = [0]

        def e2e_step():
            dsts, probb, copied, done = bufs[n_step[0] % 2]
            n_step[0] += 1
            with torch.cuda.stream(copy_stream):
                copy_stream.wait_event(done)  # the step that last used these buffers has finished with them
                for h, d in zip(step_inputs, dsts):
                    d.copy_(h, non_blocking=True)
                copied.record(copy_stream)
            stream.wait_event(copied)
            B.stepkv_compress([probb], params, ws=dt.ws, status=dt.status, stream=stream)
            done.record(stream)
            with torch.cuda.stream(stream):
                host_idx[:dt.cap].copy_(dt.out.kept_idx, non_blocking=True)
                host_idx[dt.cap:].copy_(dt.out.n_kept, non_blocking=True)

        def timed(step):
            # one untimed step first: the first transfer from freshly pinned pages runs at about a third
            # of the steady copy bandwidth
            step()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            copy_stream.wait_event(e0)
            for i in range(k2):
                step()
            e1.record(stream)
            torch.cuda.synchronize()
            return MR.max_over_ranks(e0.elapsed_time(e1) / k2, dist, dev)

        e2e_ms = timed(e2e_step)
        n_k = int(host_idx[dt.cap].item())
        assert n_k == dt.n_kept_expected
        kept_h = host_idx[:n_k].long()
        for l in (0, s_.L - 1):  # the host outputs hold the retained rows
            assert torch.equal(host_Kout[l][:, :n_k], host_K[l].index_select(1, kept_h))
            assert torch.equal(host_Vout[l][:, :n_k], host_V[l].index_select(1, kept_h))
        h2d = nb(step_inputs) + n_k * row_bytes
        d2h = n_k * row_bytes + host_idx.numel() * 4
        e2e = {"value": MR.job_throughput(tokens, e2e_ms * 1e-3), "unit": UNIT, "h2d_bytes_per_step": int(h2d),
               "d2h_bytes_per_step": int(d2h), "ms_per_step": e2e_ms, "steps": k2,
               "path": "cache in pinned host memory: window queries, token metadata, step signals and the "
                       "saliency layers' K copied to the device (two buffer sets: the next step's copies overlap "
                       "the current step's gather), retained rows gathered across the CPU-GPU link into pinned "
                       "host outputs"}

        def copy_all_step():
            for h, d in zip(host_K + host_V + host_Q + host_small, dt.K + dt.V + dt.Q + dev_small):
                d.copy_(h, non_blocking=True)
            dt.compress(params, stream)
            for h, d in zip(host_Kout + host_Vout, dt.K_out + dt.V_out):
                h.copy_(d, non_blocking=True)
            host_idx[:dt.cap].copy_(dt.out.kept_idx, non_blocking=True)
            host_idx[dt.cap:].copy_(dt.out.n_kept, non_blocking=True)

        ca_ms = timed(copy_all_step)
        assert int(host_idx[dt.cap].item()) == dt.n_kept_expected
        e2e_copy_all = {"value": MR.job_throughput(tokens, ca_ms * 1e-3), "unit": UNIT,
                        "h2d_bytes_per_step": int(nb(host_K + host_V + host_Q + host_small)),
                        "d2h_bytes_per_step": int(nb(host_Kout + host_Vout) + host_idx.numel() * 4),
                        "ms_per_step": ca_ms, "steps": k2,
                        "path": "every input copied to the device, the device pass, every output copied back"}

    # decode attention over a compacted cache (timed separately, not part of the metric): the incremental
    # loop's shape, Llama-3-8B heads, 8192-token budget + 16 prompt + 64 window rows = 8272 rows per head
    decode = None
    if rank == 0 and not args.no_decode:
        dec_rows = 8192 + 16 + 64
        dgen = torch.Generator(device=dev).manual_seed(99)
        Kd = [torch.randn((s.Hkv, dec_rows, s.d), generator=dgen, device=dev, dtype=torch.bfloat16) for _ in range(s.L)]
        Vd = [torch.randn((s.Hkv, dec_rows, s.d), generator=dgen, device=dev, dtype=torch.bfloat16) for _ in range(s.L)]
        qd = [torch.randn((s.Hq, s.d), generator=dgen, device=dev, dtype=torch.bfloat16) for _ in range(s.L)]
        outd = [torch.empty((s.Hq, s.d), dtype=torch.float32, device=dev) for _ in range(s.L)]
        ws_d = torch.empty(B.load_library().stepkv_decode_workspace_size(s.L, s.Hkv, s.Hq, s.d, dec_rows) + 512,
                           dtype=torch.uint8, device=dev)
        n_tok = 64
        for _ in range(3):
            B.stepkv_decode(qd, Kd, Vd, dec_rows, out=outd, ws=ws_d, status=dt.status, stream=stream)
        flush.fill_(7)
        torch.cuda.synchronize()
        d0, d1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        d0.record(stream)
        for _ in range(n_tok):  # the cache (1.08 GB) exceeds L2, so every token reads it from HBM
            B.stepkv_decode(qd, Kd, Vd, dec_rows, out=outd, ws=ws_d, status=dt.status, stream=stream)
        d1.record(stream)
        torch.cuda.synchronize()
        us = d0.elapsed_time(d1) * 1e3 / n_tok
        dbytes = 2 * s.L * s.Hkv * dec_rows * s.d * 2
        decode = {"workload": f"decode attention, {n_tok} single-token reads over a compacted cache of {dec_rows} "
                              f"rows x {s.L} layers x {s.Hkv} KV heads (Hq={s.Hq}, d={s.d})",
                  "us_per_token": round(us, 2), "algorithmic_bytes_per_token": dbytes,
                  "achieved_gbs": round(dbytes / (us * 1e-6) / 1e9, 1),
                  "frac_of_measured_hbm": round(dbytes / (us * 1e-6) / 1e9 / hbm, 4), "launches_per_token": 2}
        if int(dt.status.item()) != 0:
            raise RuntimeError(f"device status {int(dt.status.item())} after decode")
        del Kd, Vd

    # the incremental agent loop (timed separately, not part of the metric): Llama-3-8B heads, a 4096-token
    # start, one new step per boundary, the compacted cache plus the new step compressed under a fixed
    # 8192-token budget, then 64 single-token decode reads over the compacted cache
    incremental = None
    if rank == 0 and not args.no_incremental:
        incremental = run_incremental(args, s, dev, stream, hbm)

    clocks = sampler.stop() if sampler else None
    if dist:
        dist.barrier()
    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return

    ab = algorithmic_bytes(tr, n_kept)
    roof = None
    if stage:
        comp_gbs = ab["compact"] / (stage["compact"] * 1e-6) / 1e9
        roof = {"kernel": "compact_kernel (stage 5: retained K/V row gather, all 32 layers)", "bound": "hbm",
                "achieved": round(comp_gbs, 1), "peak": hbm, "unit": "GB/s", "frac": round(comp_gbs / hbm, 4),
                "peak_source": f"{peak_kind} hbm_gbs (burst copy)", "traffic": args.compact_traffic,
                "algorithmic_bytes_per_launch": ab["compact"], "launch_us": round(stage["compact"], 2)}
    pass_gbs = ab["total"] / (ms * 1e-3) / 1e9
    cpu = None
    if not args.no_cpu_baseline:
        secs, desc, _ = oracle_pass_seconds(args, pairs=args.oracle_pairs, compact_sets=args.oracle_compact_sets)
        cpu = {"value": s.T / secs, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": desc,
               "seconds_per_pass": round(secs, 3)}
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded generator + torch device RNG; no datasets or model weights)",
        "config": workload_config(tr, args, world),
        "roofline": roof,
        "pass_hbm": {"algorithmic_bytes": ab["total"], "achieved_gbs": round(pass_gbs, 1),
                     "frac_of_measured": round(pass_gbs / hbm, 4), "frac_of_nominal_8tbs": round(pass_gbs / 8000, 4)},
        "stages_us": {k: round(v, 2) for k, v in stage.items()} if stage else None,
        "cpu_baseline": cpu, "e2e": e2e, "e2e_copy_all": e2e_copy_all, "decode": decode, "incremental": incremental,
        "gpu_launches": launches_per_pass(tr) * args.steps,
        "clocks": clocks,
        "wall_s_timed_region": round(wall1 - wall0, 4),
        "step_ms_min_max": [round(min(step_ms), 4), round(max(step_ms), 4)],
        "n_kept": n_kept,
    }
    print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()


def run_incremental(args, s, dev, stream, hbm):
    """Boundaries of the incremental loop on device-random K/V/Q (layout and signals from the seeded
    generator).  The cache lives in one capacity buffer per layer and is compacted in place (hole
    filling); each new step is appended after the retained rows.  Events time each compression and each
    group of 64 decode reads."""
    import numpy as np
    import torch
    from paper_2609_22158_gb300 import binding as B, workload as wl
    budget, t0, n_dec = 8192, 4096, 64
    lp = wl.IncrementalLoop(5, L=s.L, Hq=s.Hq, Hkv=s.Hkv, d=s.d, W=s.W, t0=t0, budget_count=budget)
    gen = torch.Generator(device=dev).manual_seed(55)
    cap = budget + 16 + 4 * s.W + 2400  # retained rows + the largest new step
    Kbuf = [torch.randn((s.Hkv, cap, s.d), generator=gen, device=dev, dtype=torch.bfloat16) for _ in range(s.L)]
    Vbuf = [torch.randn((s.Hkv, cap, s.d), generator=gen, device=dev, dtype=torch.bfloat16) for _ in range(s.L)]
    step_id, n_steps = lp.initial_layout()
    pos = np.arange(t0, dtype=np.int32)
    next_pos = t0
    reuse = np.zeros(n_steps, np.float32)
    params = B.Params()
    status = B.new_status(dev)
    comp_us, dec_us, rows, moved = [], [], [], []
    ws = torch.empty(64 << 20, dtype=torch.uint8, device=dev)
    ws_d = torch.empty(B.load_library().stepkv_decode_workspace_size(s.L, s.Hkv, s.Hq, s.d, cap) + 512,
                       dtype=torch.uint8, device=dev)
    outd = [torch.empty((s.Hq, s.d), dtype=torch.float32, device=dev) for _ in range(s.L)]
    for b in range(args.inc_boundaries):
        if b > 0:
            n_new = lp.step_length(b)
            n_steps += 1
            T0 = int(step_id.shape[0])
            if T0 + n_new > cap:
                raise RuntimeError("capacity buffer too small")
            for k, v in zip(Kbuf, Vbuf):  # the new step's rows, after the retained ones
                k[:, T0:T0 + n_new].normal_(generator=gen)
                v[:, T0:T0 + n_new].normal_(generator=gen)
            step_id = np.concatenate([step_id, np.full(n_new, n_steps - 1, np.int32)])
            pos = np.concatenate([pos, np.arange(next_pos, next_pos + n_new, dtype=np.int32)])
            next_pos += n_new
            reuse = np.concatenate([reuse, np.float32([0.0])])
        T = int(step_id.shape[0])
        prot = lp.protected(step_id)
        valid, gain, red, obs_sim = lp.signals(b, n_steps)
        t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
        reuse_out = torch.empty(n_steps, dtype=torch.float32, device=dev)
        steps = B.StepSignals(t(valid), t(gain), t(red), t(reuse), t(obs_sim), reuse_out)
        kcap = min(T, budget + int(prot.sum()))
        out = B.SelectOutputs.allocate(T, n_steps, kcap, dev, full=False)
        sid_out = torch.empty(kcap, dtype=torch.int32, device=dev)
        pos_out = torch.empty(kcap, dtype=torch.int32, device=dev)
        Q = [torch.randn((s.Hq, s.W, s.d), generator=gen, device=dev, dtype=torch.bfloat16) for _ in range(s.Ls)]
        live_K = [k[:, :T] for k in Kbuf]
        live_V = [v[:, :T] for v in Vbuf]
        prob = B.Problem(live_K, live_V, Q, T, t(step_id), t(prot), steps, B.budget_count(budget), live_K, live_V,
                         out, pos_in=t(pos), step_id_out=sid_out, pos_out=pos_out)
        need = B.stepkv_workspace_size([prob])
        assert need <= ws.numel() - 512
        qd = [torch.randn((s.Hq, s.d), generator=gen, device=dev, dtype=torch.bfloat16) for _ in range(s.L)]
        torch.cuda.synchronize()
        torch.cuda._sleep(300_000)  # the device stays busy while the host prepares the call
        e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
        e[0].record(stream)
        B.stepkv_compress([prob], params, ws=ws, status=status, stream=stream)
        e[1].record(stream)
        for _ in range(n_dec):
            B.stepkv_decode(qd, live_K, live_V, out.n_kept, out=outd, ws=ws_d, status=status, stream=stream)
        e[2].record(stream)
        torch.cuda.synchronize()
        if int(status.item()) != 0:
            raise RuntimeError(f"device status {int(status.item())} at boundary {b}")
        n = int(out.n_kept.item())
        kept = out.kept_idx[:n].cpu().numpy()
        rows.append(T)
        moved.append(int((kept >= n).sum()))
        comp_us.append(e[0].elapsed_time(e[1]) * 1e3)
        dec_us.append(e[1].elapsed_time(e[2]) * 1e3 / n_dec)
        step_id = sid_out[:n].cpu().numpy()
        pos = pos_out[:n].cpu().numpy()
        reuse = reuse_out.cpu().numpy()
    steady = [i for i in range(len(rows)) if rows[i] > budget + 2 * s.W]  # the budget binds
    pick = steady or list(range(len(rows)))
    mean = lambda xs: float(np.mean([xs[i] for i in pick]))
    return {"workload": f"incremental loop: {args.inc_boundaries} boundaries from a {t0}-token start, one new "
                        f"step each, fixed {budget}-token budget, cache compacted in place (hole filling), "
                        f"{n_dec} decode reads after each compression; {s.L} layers, Hq={s.Hq}, Hkv={s.Hkv}, "
                        f"d={s.d}, W={s.W}",
            "boundaries_with_budget_binding": len(steady),
            "cache_rows_mean": round(mean(rows), 1), "rows_moved_mean": round(mean(moved), 1),
            "compress_us_mean": round(mean(comp_us), 2),
            "decode_us_per_token_mean": round(mean(dec_us), 2),
            "compress_tokens_per_s": round(mean(rows) / (mean(comp_us) * 1e-6))}


# ---------------------------------------------------------------------------------- reference arm
def run_reference(args):
    """The oracle as it stands on the host cores, same workload/metric; each step a bounded sample."""
    from paper_2609_22158_gb300 import multirank as MR
    world, rank, _ = MR.rank_env()
    if rank != 0:
        return
    tr = make_traj(args)
    s = tr.shape
    times = []
    desc = ""
    for i in range(args.warmup + args.steps):
        secs, desc, _ = oracle_pass_seconds(args, pairs=args.ref_pairs, compact_sets=args.ref_compact_sets)
        if i >= args.warmup:
            times.append(secs)
    sec = sum(times) / len(times)
    value = s.T / sec
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic (seeded generator)",
        "config": workload_config(tr, args, 1),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": desc},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--seed", type=int, default=1)
    ap.add_argument("--T", type=int, default=32768)
    ap.add_argument("--layers", type=int, default=32)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=8)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-stages", action="store_true")
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--no-incremental", action="store_true")
    ap.add_argument("--inc-boundaries", type=int, default=24)
    ap.add_argument("--oracle-pairs", type=int, default=24)
    ap.add_argument("--oracle-compact-sets", type=int, default=16)
    ap.add_argument("--ref-pairs", type=int, default=2)
    ap.add_argument("--ref-compact-sets", type=int, default=4)
    ap.add_argument("--compact-traffic", type=float, default=None,
                    help="dram bytes (read+write) per compaction launch from an ncu capture of this workload "
                         "(default: the capture of the current compaction kernel for the 32-layer 32K workload)")
    args = ap.parse_args()
    if args.compact_traffic is None and args.T == 32768 and args.layers == 32:
        # dram__bytes_read.sum + dram__bytes_write.sum of compact_kernel from one single-pass ncu capture
        # of this workload at full size (the timed step's launch): 438.94 MB read + 388.77 MB written.
        # The ~50 MB of writes below the algorithmic bytes are dirty lines still in L2 when it ends.
        args.compact_traffic = 438.94e6 + 388.77e6
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
