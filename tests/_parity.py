"""Shared helpers of the GPU parity tests (GPU path vs CPU oracle).

Comparison rules:
* loop counts and active sets: bit-exact for every token whose router margin
  (from the oracle's depth table) exceeds 1e-3; near-tie tokens are forced to
  the oracle's loop count on both sides and counted;
* logits: per row max |gpu - oracle| / max |oracle| <= tol (2e-2 for bf16
  models, 1e-4 for float32 models); the worst row is returned.
"""
import numpy as np

from oracle import tlf_oracle as O

NEAR_TIE = 1e-3


def tol_for(model):
    return 1e-4 if model.dtype == "f32" else 2e-2


def rel_err(g, o):
    g = np.atleast_2d(np.asarray(g, dtype=np.float64))
    o = np.atleast_2d(np.asarray(o, dtype=np.float64))
    return float(np.max(np.max(np.abs(g - o), axis=1) / np.max(np.abs(o), axis=1)))


class DepthOracle:
    """Depth table of every token id plus the near-tie forcing rule."""

    def __init__(self, omodel):
        self.table, self.margin = O.depth_table(omodel)
        self.near = self.margin <= NEAR_TIE
        self.n_forced = 0

    def forced_for(self, tokens):
        t = np.asarray(tokens)
        f = np.where(self.near[t], self.table[t], -1).astype(np.int32)
        self.n_forced += int((f > 0).sum())
        return f

    def expected(self, tokens, forced=None):
        m = self.table[np.asarray(tokens)].astype(np.int32)
        if forced is not None:
            m = np.where(np.asarray(forced) >= 1, forced, m)
        return m


def check_active_sets(ctx, loops, M):
    counts, sets = ctx.last_active_sets(len(loops))
    for r in range(M):
        want = np.nonzero(loops >= r + 1)[0]
        assert counts[r] == want.size, (r, counts[r], want.size)
        np.testing.assert_array_equal(sets[r], want)


def check_cache(ctx, seq_id, oseq, model, tol):
    """GPU cache of one sequence against the oracle's: positions exact, K/V within tol."""
    for i in range(model.max_loops):
        for j in range(model.n_layers):
            gp, gk, gv = ctx.read_cache(seq_id, i + 1, j)
            op, ok, ov = oseq.caches[i][j].view()
            np.testing.assert_array_equal(gp, op)
            if len(op):
                assert rel_err(gk.reshape(len(op), -1), ok.reshape(len(op), -1)) < tol
                assert rel_err(gv.reshape(len(op), -1), ov.reshape(len(op), -1)) < tol
