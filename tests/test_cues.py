"""Host-side evidence cues (the library's reference reading of Sec. 4.1's cue extraction): CPU only."""
import numpy as np

from oracle import stepkv_oracle as O
from paper_2609_22158_gb300 import cues as C, workload as wl


def test_text_cues_are_sorted_distinct_and_capped():
    a = C.text_cues("The tool returned 3 results: Paris, paris, Lyon and the Rhone river in France.")
    assert a.dtype == np.uint32 and np.all(np.diff(a.astype(np.int64)) > 0)
    assert len(a) == len(set(["returned", "3", "results", "paris", "lyon", "rhone", "river", "france", "tool"]))
    long = " ".join(f"word{i}" for i in range(200))
    assert len(C.text_cues(long)) == 64
    assert np.array_equal(C.text_cues("Paris Lyon"), C.text_cues("lyon, PARIS"))


def test_cue_overlap_follows_shared_words():
    a, b = C.text_cues("capital city of France is Paris"), C.text_cues("Paris is the capital city of France")
    c = C.text_cues("Tokyo population statistics")
    assert O.cue_similarity(a, b) == 1.0 and O.cue_similarity(a, c) == 0.0


def test_observation_validity():
    assert C.observation_valid("Paris is the capital") == 1.0
    assert C.observation_valid("   ") == 0.0
    assert C.observation_valid("Error: tool timed out") == 0.0


def test_pack_and_synthetic_cues():
    steps = wl.synthetic_cues(3, 12)
    cues, cnt = C.pack_cues(steps)
    assert cues.shape == (12, 3, 64) and cnt.shape == (12, 3)
    for k in range(12):
        for f in range(3):
            v = cues[k, f, :cnt[k, f]].astype(np.int64)
            assert np.all(np.diff(v) > 0) and np.array_equal(v, np.asarray(steps[k][f], np.int64))
    gain, red, obs_sim = O.step_signals([s[0] for s in steps], [s[1] for s in steps], [s[2] for s in steps], k0=0)
    assert (red[1:] > 0).any() and (obs_sim[:-1] > 0).any() and (gain < 1).any()
