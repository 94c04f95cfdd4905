"""The oracle's step 1 (Sec. 3.3, C_i = TopK(q_i, K), and the log-partition) over every row of
a full-size logit tensor, spread over the host cores.

A full stable sort of one 126464-entry row takes tens of milliseconds in the oracle, so the
4096 rows of a full-size block run in a pool of fresh interpreters (started with `spawn`: a
process forked from one that has used CUDA can hang). The workers import only numpy and the
oracle; rows reach them as float32 arrays, an exact widening of bf16 or fp32 logits.
"""
from __future__ import annotations

import multiprocessing as mp
import os
from concurrent.futures import ProcessPoolExecutor

import numpy as np

ROWS_PER_TASK = 32


def _topk_rows(rows: np.ndarray, K: int):
    from oracle import brisk_oracle as O
    n = rows.shape[0]
    ids = np.zeros((n, K), np.int64)
    lp = np.zeros((n, K))
    lse = np.zeros(n)
    for j in range(n):
        ids[j], lp[j], lse[j] = O.topk_candidates(rows[j].astype(np.float64), K)
    return ids, lp, lse


def topk_all_rows(rows: np.ndarray, K: int, workers: int = 0):
    """Oracle candidates of every row of `rows` [N, V] (float32): ids [N, K], log-probs [N, K]
    and log-partitions [N], in row order."""
    rows = np.ascontiguousarray(rows, dtype=np.float32)
    n = rows.shape[0]
    if workers <= 0:
        workers = max(1, min(16, len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity")
                             else (os.cpu_count() or 1)))
    starts = list(range(0, n, ROWS_PER_TASK))
    with ProcessPoolExecutor(max_workers=workers, mp_context=mp.get_context("spawn")) as ex:
        parts = list(ex.map(_topk_rows, [rows[s:s + ROWS_PER_TASK] for s in starts],
                            [K] * len(starts)))
    return (np.concatenate([p[0] for p in parts]), np.concatenate([p[1] for p in parts]),
            np.concatenate([p[2] for p in parts]))
