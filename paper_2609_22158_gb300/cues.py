"""Evidence cues of a step's fields, for stepkv_step_signals (Sec. 4.1: field similarity is the overlap of up
to 64 evidence cues per field).  The paper does not say how cues are drawn from text; this module is the
library's reference reading, host-side preprocessing that callers may replace: the distinct content words and
numbers of a field (lower-cased alphanumeric runs of 3 or more characters, or any number, minus a short
stop-word list), each hashed to 32 bits (FNV-1a), the first 64 distinct ones in order of appearance, returned
sorted as the kernel expects.  An Observation is unusable (valid = 0) when it is empty or reports an error.
"""
from __future__ import annotations

import re
from typing import Iterable, List, Sequence, Tuple

import numpy as np

MAX_CUES = 64  # STEPKV_MAX_CUES
_STOP = frozenset("""the and for are but not you all any can had her was one our out has have him his how its
may new now see two who did get let man put say she too use with that this from they will would there their
what about which when were been into than then them these some could other only also more most such very just
over your yours each here where while""".split())
_WORD = re.compile(r"[a-z0-9]+")
_ERROR = re.compile(r"^\s*(error|exception|traceback|failed|failure|no results?)\b", re.IGNORECASE)


def _fnv1a32(s: str) -> int:
    h = 0x811C9DC5
    for b in s.encode("utf-8"):
        h ^= b
        h = (h * 0x01000193) & 0xFFFFFFFF
    return h


def text_cues(text: str, cap: int = MAX_CUES) -> np.ndarray:
    """Sorted distinct uint32 cue ids of one field's text (at most ``cap``)."""
    seen, out = set(), []
    for w in _WORD.findall(text.lower()):
        if (len(w) < 3 and not w.isdigit()) or w in _STOP:
            continue
        h = _fnv1a32(w)
        if h in seen:
            continue
        seen.add(h)
        out.append(h)
        if len(out) == cap:
            break
    return np.array(sorted(out), dtype=np.uint32)


def observation_valid(text: str) -> float:
    """valid_k of Eq. 2: 0 for an empty or error-returning Observation, else 1."""
    return 0.0 if (not text.strip() or _ERROR.match(text)) else 1.0


def pack_cues(fields: Sequence[Tuple[Iterable[int], Iterable[int], Iterable[int]]]):
    """Per step (Thought, Action, Observation) cue lists -> (cues [n_steps, 3, 64] uint32, n_cues [n_steps, 3]
    int32), the layout of stepkv_step_signals."""
    n = len(fields)
    cues = np.zeros((n, 3, MAX_CUES), dtype=np.uint32)
    cnt = np.zeros((n, 3), dtype=np.int32)
    for k, fs in enumerate(fields):
        for f, lst in enumerate(fs):
            a = np.unique(np.asarray(list(lst), dtype=np.uint32))[:MAX_CUES]
            cues[k, f, :len(a)] = a
            cnt[k, f] = len(a)
    return cues, cnt
