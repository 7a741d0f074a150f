"""Simulator of the mask recurrence of Algorithm 1 (App. E.1), written from the paper's text.

It is independent of the oracle: it never evaluates the ancestor rule directly. It runs the
logical fused decoding loop over one page:

  * prefill of X (the image/prompt prefix), causal inside X;
  * every iteration appends one input per live stream to the cache, and each stream's mask row
    gains exactly its own new position (the identity block, M <- [M I_C]);
  * when the layout stream has put f_k tokens in the cache, branch k is created with a copy of the
    layout stream's current row (the pre-boundary row), and starts appending on the next
    iteration;
  * a stream retires after its last token (the layout stream after L tokens, branch k after n_k).

It returns, for every token, the set of tokens visible to it when it was decoded, expressed in
page-local packed positions [X | layout | Y_1 | ... | Y_N].
"""
from __future__ import annotations

import numpy as np


def simulate(P, L, forks, lens):
    N = len(lens)
    ybase = [P + L + sum(lens[:k]) for k in range(N)]
    S = P + L + sum(lens)
    vis = np.zeros((S, S), np.uint8)
    # cache positions are labelled directly with their packed position
    # prefill of X: causal inside the prefix
    for i in range(P):
        vis[i, : i + 1] = 1
    layout_row = set(range(P))   # the layout stream's row before it appends anything
    layout_count = 0
    child_rows = {}              # branch -> current row
    child_done = {}              # branch -> tokens appended so far
    pending = [k for k in range(N)]

    def fork_ready():
        for k in list(pending):
            if forks[k] == layout_count:
                child_rows[k] = set(layout_row)   # copy of the pre-boundary row
                child_done[k] = 0
                pending.remove(k)

    fork_ready()
    live = True
    while live:
        appended = False
        # one input per live stream: the identity block gives each stream its own new position
        if layout_count < L:
            pos = P + layout_count
            layout_row.add(pos)
            for j in layout_row:
                vis[pos, j] = 1
            layout_count += 1
            appended = True
        for k in sorted(child_rows):
            if child_done[k] < lens[k]:
                pos = ybase[k] + child_done[k]
                child_rows[k].add(pos)
                for j in child_rows[k]:
                    vis[pos, j] = 1
                child_done[k] += 1
                appended = True
        fork_ready()
        live = appended or bool(pending)
        if not appended and pending:
            raise RuntimeError("fork offset beyond the layout stream")
    return vis
