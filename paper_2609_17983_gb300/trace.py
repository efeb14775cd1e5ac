"""Device timeline of a traced pass (records from Model.trace_read()).

Every CTA of the pass kernels leaves one record: kind, SM, block index, the
time it started, the time its wait on the predecessor kernel returned, the
time it finished, and eight kernel-specific marks (GEMM, for the CTA's last
tile: first operand stage landed, all MMAs complete, accumulator taken by the
epilogue, partial stored, split-tile arrival counted or partials staged across
the cluster, tile reduced and written, epilogue done, all warps done;
attention: last key chunk consumed; Attention-selector logits: keys and
queries staged, logits computed, chunk statistics stored, arrival counted,
fold done).  `launches` groups the records into kernel launches
(a launch holds each block index once), in issue order; `layer_table`
averages the launches of a repeating per-layer sequence by position.
"""
from __future__ import annotations

import numpy as np

KINDS = {1: "embed", 2: "rmsnorm", 3: "gemm", 4: "rope", 5: "attention", 6: "combine", 7: "other",
         8: "select", 9: "select_accum"}


def launches(rec: np.ndarray) -> list[dict]:
    rec = np.asarray(rec, np.uint64)
    out = []
    for kind in np.unique(rec[:, 0] & np.uint64(0xFF)):
        r = rec[(rec[:, 0] & np.uint64(0xFF)) == kind]
        r = r[np.argsort(r[:, 1], kind="stable")]
        blocks = (r[:, 0] >> np.uint64(16)).astype(np.int64)
        cur, seen = [], set()
        groups = []
        for i, b in enumerate(blocks):
            if b in seen:
                groups.append(cur)
                cur, seen = [], set()
            cur.append(i)
            seen.add(b)
        if cur:
            groups.append(cur)
        for g in groups:
            t = r[g, 1:12].astype(np.int64)
            d = dict(kind=KINDS.get(int(kind), str(int(kind))), ctas=len(g),
                     start=int(t[:, 0].min()), wait=int(np.median(t[:, 1])),
                     wait_last=int(t[:, 1].max()), end=int(t[:, 2].max()),
                     end_median=int(np.median(t[:, 2])))
            for k in range(8):
                mk = t[:, 3 + k][t[:, 3 + k] > 0]
                d[f"mark{k}"] = int(np.median(mk)) if len(mk) else 0
                d[f"mark{k}_last"] = int(mk.max()) if len(mk) else 0
            out.append(d)
    out.sort(key=lambda x: x["start"])
    return out


def layer_table(ls: list[dict], pattern: list[str], names: list[str] | None = None) -> list[dict]:
    """Average, over repeats of `pattern` (kinds in order), of each position:
    time from the previous launch's last end to this launch's median wait
    return (dependency latency), and from that to its last end (run)."""
    names = names or pattern
    kinds = [x["kind"] for x in ls]
    starts = [i for i in range(len(ls) - len(pattern) + 1) if kinds[i:i + len(pattern)] == pattern]
    rows = []
    for j, nm in enumerate(names):
        lat, run, span = [], [], []
        for i in starts:
            x = ls[i + j]
            prev = ls[i + j - 1] if i + j > 0 else None
            if prev is not None:
                lat.append(x["wait"] - prev["end"])
            run.append(x["end"] - x["wait"])
            span.append(x["end"] - (prev["end"] if prev is not None else x["start"]))
        rows.append(dict(name=nm, repeats=len(starts), latency_us=np.mean(lat) / 1e3 if lat else 0.0,
                         run_us=np.mean(run) / 1e3, span_us=np.mean(span) / 1e3))
    return rows
