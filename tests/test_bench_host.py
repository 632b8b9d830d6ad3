"""Host-side arithmetic of bench.py that the reported roofline fractions and launch counts rest on, checked
against counts written out from the workload's shapes (no GPU)."""
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

import bench  # noqa: E402
from paper_2609_22158_gb300 import workload as wl  # noqa: E402


def test_config2_algorithmic_bytes():
    """The 32K workload's minimum bytes per pass, stage by stage: the saliency reads the 3 saliency layers'
    keys (8 KV heads x 32768 rows x 256 B) and the window queries (32 heads x 64 rows x 256 B) and writes
    one fp32 per (layer, KV head, token); the selection reads those and the step id and mask per token and
    writes the retained slots; the compaction reads and writes every retained row of K and V in all 32
    layers and 8 KV heads, plus three int32 per retained row (index, step id, position)."""
    tr = bench.make_trajs(2)[0]
    s = tr.shape
    assert (s.L, s.Hq, s.Hkv, s.d, s.T, s.W, s.Ls) == (32, 32, 8, 128, 32768, 64, 3)
    n_kept = 3348
    ab = bench.algorithmic_bytes(tr, n_kept)
    keys = 3 * 8 * 32768 * 256          # 201,326,592
    queries = 3 * 32 * 64 * 256         # 1,572,864
    sal = 3 * 8 * 32768 * 4             # 3,145,728
    assert ab["score"] == keys + queries + sal == 206045184
    assert ab["select"] == sal + 32768 * (4 + 1) + n_kept * 4 == 3322960
    rows = n_kept * 32 * 8 * 2          # retained rows of K and V over all layers and KV heads
    assert ab["compact"] == rows * 256 * 2 + n_kept * 12 == 877698288
    assert ab["total"] == 1087066432
    # one pass of the contraction: 2 flop per (layer, query head, window row, key, channel)
    assert ab["score_flops_one_pass"] == 2.0 * 3 * 32 * 64 * 32768 * 128
    assert ab["score_exps_one_pass"] == 3.0 * 32 * 64 * 32768


def test_launches_per_call():
    """Launches of one stepkv_compress call: a saliency launch per batch of up to 16 trajectories and 512 MB
    of saliency keys, a selection launch per 16 trajectories, and compaction launches of up to 16
    trajectories and 1024 (layer, tensor) entries."""
    assert bench.launches_per_call(bench.make_trajs(2)) == 3
    small = [wl.custom(i, L=2, Hq=4, Hkv=2, d=64, T=400, W=16, n_steps=3) for i in range(20)]
    assert bench.launches_per_call(small) == 2 + 2 + 2
    # 300 layers x K and V = 600 entries per trajectory: two trajectories need two compaction launches
    big = [wl.custom(i, L=300, Hq=4, Hkv=2, d=64, T=400, W=16, n_steps=3) for i in range(2)]
    assert bench.launches_per_call(big) == 1 + 1 + 2


def test_traffic_constants_cover_the_config2_kernels():
    """The DRAM traffic quoted beside the roofline comes from a capture of each of the pass's kernels."""
    t = bench.NCU_TRAFFIC[2]
    assert set(t) == {"score_kernel", "select_kernel", "compact_kernel"}
    assert all(v > 0 for v in t.values())
