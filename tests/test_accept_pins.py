"""Pins for the oracle's bifurcation test (Algorithm 1): accept counts from
top-beta ranks of the drafted bytes. Each test reaches the count by a
different route than the oracle's strictly-larger count: argmax for beta = 1,
a full descending sort, or hand-built rows."""
import numpy as np

import oracle

RNG = np.random.default_rng(2024)


def test_beta_one_is_greedy_argmax():
    streams, k = 6, 9
    logits = RNG.standard_normal((streams, k, 256))   # distinct values almost surely
    best = logits.argmax(axis=2)
    drafted = best.copy()
    cut = [0, 3, 9, 1, 5, 8]
    for s, c in enumerate(cut):
        if c < k:
            drafted[s, c] = (best[s, c] + 1) % 256      # first non-greedy byte at c
    assert oracle.accept_topk(logits, drafted, 1).tolist() == [min(c, k) for c in cut]


def test_rank_from_a_full_sort():
    streams, k, beta = 5, 7, 17
    logits = np.round(RNG.standard_normal((streams, k, 256)), 1)   # many ties
    drafted = RNG.integers(0, 256, (streams, k))
    want = []
    for s in range(streams):
        a = k
        for i in range(k):
            desc = np.sort(logits[s, i])[::-1]
            rank = int(np.argmax(desc == logits[s, i, drafted[s, i]])) + 1   # first occurrence
            if rank > beta:
                a = i
                break
        want.append(a)
    assert oracle.accept_topk(logits, drafted, beta).tolist() == want


def test_ties_share_the_better_rank_and_edges():
    row = np.zeros(256)
    row[[3, 7]] = 5.0                      # two equal maxima: both rank 1
    row[9] = 4.0                           # rank 3
    logits = np.tile(row, (1, 3, 1))
    assert oracle.accept_topk(logits, np.array([[7, 3, 9]]), 1).tolist() == [2]
    assert oracle.accept_topk(logits, np.array([[7, 3, 9]]), 3).tolist() == [3]
    assert oracle.accept_topk(logits, np.array([[0, 3, 9]]), 3).tolist() == [0]   # rank 4
    assert oracle.accept_topk(logits, np.array([[0, 0, 0]]), 256).tolist() == [3]  # beta = vocab
    assert oracle.accept_topk(np.zeros((2, 0, 256)), np.zeros((2, 0), dtype=int), 1).tolist() == [0, 0]
