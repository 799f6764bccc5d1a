"""The synthetic workloads' loop-count distributions (long-tailed, Fig. 1b) as the oracle routes them.

With rotary positions and no absolute position embedding the router reads
RMSNorm(E[x]) only, so a token's loop count is a function of its id and the
distribution over the vocabulary is the distribution of any long run of
uniform random tokens. The router bias is fitted (in synth) against Gaussian
draws with the router's covariance, never by routing tokens; these tests pin
what the oracle's router then gives over every id of the vocabulary:
the histogram of the depth table matches the stated target within 0.01 per
loop count, and the mean depth matches the target's (C4: 3.70; the paper
reports 3.69 for FineWeb-Edu, Fig. 1b).
"""
import functools

import numpy as np
import pytest

from oracle import tlf_oracle as O
from paper_2609_15160_gb300 import synth


@functools.lru_cache(maxsize=None)
def _depth_table(name):
    m = synth.get_config(name).model
    return m, O.depth_table(O.OracleModel.from_config(m, synth.make_weights(m)))


@pytest.mark.parametrize("name", ["c2", "c3", "c4"])
def test_depth_table_matches_the_target_distribution(name):
    m, (table, margin) = _depth_table(name)
    assert table.shape == (m.vocab,) and table.min() >= 1 and table.max() <= m.max_loops
    hist = np.bincount(table, minlength=m.max_loops + 1)[1:] / m.vocab
    target = np.asarray(m.depth_probs)
    assert np.max(np.abs(hist - target)) < 0.01, (hist.round(4), target)
    mean = float(np.sum(hist * np.arange(1, m.max_loops + 1)))
    assert abs(mean - synth.expected_mean_depth(target)) < 0.03, mean
    # the tail the paper describes: the deepest loop count is reached by some but few tokens
    assert 0 < hist[-1] < hist.max()
    # near-tie ids (margin <= 1e-3) are a small minority, so bit-exact loop counts cover almost all ids
    assert np.mean(margin <= 1e-3) < 0.01


def test_c4_mean_depth_is_the_papers():
    _, (table, _) = _depth_table("c4")
    assert abs(float(table.mean()) - 3.69) < 0.02
