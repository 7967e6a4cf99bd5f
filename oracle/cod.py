"""Conditional drop-token (COD) data construction -- oracle (test
infrastructure only).

Follows Section 3.2 ("Mask Tokens based Training", "Conditional Drop of
Tokens") and the appendix algorithm and worked example of the paper:

* A training sample of N+1 tokens x_0..x_N is split into K subtasks.
  Subtask 1 is ordinary next-token training: the row at position j feeds x_j
  and is labelled x_{j+1} (j = 0..N-1).  Subtask k >= 2 predicts the k-th next
  token: its row at position j feeds the mask token m_{k-2} and is labelled
  x_{j+1}; it attends to the real rows at positions 0..j-k+1 and to the
  subtask rows k' = 2..k-1 at positions j-k+k' (one mask of each earlier
  mask subtask, the chain the loss of subtask k conditions on), and to itself.
  Its rows exist for j = k-2..N-1 (the chain starts at a subtask-2 row).
* Retention: subtask k keeps n_k = round(N * max(r^(k-1), r_min)) rows
  (r^(k-1) by repeated multiplication in double, round half up).
* Integrity of prefix key-value states: a row of subtask k >= 3 is a
  candidate only if its predecessor (subtask k-1, position j-1) was kept, so
  every kept row finds its whole attention context.  Subtask 2 rows only
  need real rows and are all candidates.
* Among the candidates, n_k are chosen at random (all of them when there are
  fewer): here the candidates with the n_k smallest Philox words (stream 3,
  step = sample id, sequence 0, row k, v = j), ties to the lower j.

Subtask 1 keeps every row.  The result is the keep flags of subtasks
2..K; the packed training data (input ids, labels, positions, the attention
chain) follows from them by bookkeeping (``packed_rows``).
"""
from __future__ import annotations

from typing import List, Sequence, Tuple

import numpy as np

from .philox import raw_words

STREAM_COD = 3


def retained_count(N: int, k: int, r: float, r_min: float) -> int:
    """n_k = round(N * max(r^(k-1), r_min)), half up, in double."""
    g = 1.0
    for _ in range(k - 1):
        g *= float(r)
    g = max(g, float(r_min))
    return int(np.floor(N * g + 0.5))


def cod_select(N: int, K: int, r: float, r_min: float, seed: int, sample_id: int,
               forced: Sequence[Sequence[int]] = ()) -> Tuple[np.ndarray, List[int]]:
    """Keep flags [K-1][N] for subtasks 2..K (row j of subtask k at index
    [k-2][j]) and the number of rows kept per subtask 1..K.  forced[k-2], if
    given, lists the positions subtask k keeps instead of the random choice
    (for replaying the paper's worked example)."""
    keep = np.zeros((max(K - 1, 0), N), dtype=np.int32)
    counts = [N]
    for k in range(2, K + 1):
        cand = []
        for j in range(k - 2, N):
            if k == 2 or keep[k - 3, j - 1] == 1:
                cand.append(j)
        n = retained_count(N, k, r, r_min)
        if k - 2 < len(forced):
            chosen = [int(j) for j in forced[k - 2]]
            assert all(j in cand for j in chosen), "forced choice outside the candidates"
        else:
            if cand:
                w = raw_words(seed, STREAM_COD, sample_id, 0, k, np.asarray(cand, dtype=np.uint64))
                order = sorted(range(len(cand)), key=lambda t: (int(w[t]), cand[t]))
                chosen = [cand[t] for t in order[:n]]
            else:
                chosen = []
        for j in chosen:
            keep[k - 2, j] = 1
        counts.append(len(chosen))
    return keep, counts


def candidates(keep: np.ndarray, k: int, N: int) -> List[int]:
    """Rows of subtask k whose attention chain is complete given keep."""
    return [j for j in range(k - 2, N) if k == 2 or keep[k - 3, j - 1] == 1]


def packed_rows(tokens: Sequence[int], keep: np.ndarray, mask_ids: Sequence[int]):
    """The processed sample: one tuple per row, subtask by subtask,
    (subtask k, input id, position, label, index of the predecessor row in
    this list or -1, number of real rows attended)."""
    N = len(tokens) - 1
    K = keep.shape[0] + 1
    rows, where = [], {}
    for j in range(N):
        where[(1, j)] = len(rows)
        rows.append((1, int(tokens[j]), j, int(tokens[j + 1]), -1, j + 1))
    for k in range(2, K + 1):
        for j in range(N):
            if keep[k - 2, j]:
                prev = where[(k - 1, j - 1)] if k >= 3 else -1
                where[(k, j)] = len(rows)
                rows.append((k, int(mask_ids[k - 2]), j, int(tokens[j + 1]), prev, max(j - k + 2, 0)))
    return rows
