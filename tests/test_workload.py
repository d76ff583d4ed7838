"""The synthetic input generator: determinism and distributions (no GPU)."""
import math

import numpy as np
import torch

from oracle import oracle as O
from paper_2205_11048_gb300 import workload as W


def test_deterministic_and_shapes():
    c = W.reduced(3)
    a = W.generate_step(c, 2, "cpu")
    b = W.generate_step(c, 2, "cpu")
    assert len(a) == c.M
    for x, y in zip(a, b):
        assert x["token"] == y["token"]
        for t in range(len(c.tables)):
            assert torch.equal(x["ids"][t], y["ids"][t])
            assert torch.equal(x["rows"][t], y["rows"][t])
            assert x["rows"][t].shape == (x["ids"][t].numel(), c.tables[t].dim)
            assert x["ids"][t].numel() <= c.max_ids_per_msg(t)
            assert int(x["ids"][t].min()) >= 0 and int(x["ids"][t].max()) < c.tables[t].rows
        assert torch.equal(x["dense"], y["dense"])


def test_zipf_matches_law():
    g = torch.Generator().manual_seed(1)
    r = W.zipf_ranks(1_000_000, 5000, 1.05, g, "cpu")
    assert int(r.min()) >= 1 and int(r.max()) <= 5000
    H = sum(k ** -1.05 for k in range(1, 5001))
    for k in (1, 2, 5, 50):
        p = k ** -1.05 / H
        f = float((r == k).double().mean())
        assert abs(f - p) < 5 * math.sqrt(p / 1e6) + 1e-4


def test_hash64_is_splitmix64():
    xs = [0, 1, 12345, 2**63 - 1, -1, -(2**62)]
    got = W.hash64(torch.tensor(xs, dtype=torch.int64)).tolist()
    for x, v in zip(xs, got):
        assert (v & (2**64 - 1)) == O.splitmix64(x & (2**64 - 1))


def test_staleness_distributions():
    cfg = W.config(2)
    s = []
    for k in range(400):
        toks = W.tokens_for_step(cfg, 1000 + k)
        s += [1000 + k - t for t in toks]
    s = np.array(s)
    strag = (s >= 5).mean()
    assert 0.07 < strag < 0.14
    assert s.max() <= 20 and s.min() >= 0
    cfg4 = W.config(4)
    s4 = np.array([1000 - t for k in range(300) for t in W.tokens_for_step(cfg4, 1000)])
    assert s4.max() <= 50
    assert W.tokens_for_step(W.config(1), 7) == [7, 7, 7, 7]
    # tokens never negative
    assert min(W.tokens_for_step(cfg, 0)) == 0
