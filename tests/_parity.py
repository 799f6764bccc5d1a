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


def check_active_sets(ctx, loops, M, ablation="none"):
    """The rows each loop ran on: A_r = {b : m_b >= r} in increasing b (Eq. 4-6).

    Without the gather (the no-gather ablation) every loop that has an active
    token lists all rows of the step instead.
    """
    counts, sets = ctx.last_active_sets(len(loops))
    for r in range(M):
        want = np.nonzero(loops >= r + 1)[0]
        if ablation == "no_gather" and want.size:
            want = np.arange(len(loops))
        assert counts[r] == want.size, (r, counts[r], want.size)
        np.testing.assert_array_equal(sets[r], want)


def cache_tol(model, prefilled=True):
    """Tolerance of a stored K/V entry row (max abs diff / row max).

    An entry of loop i is an intermediate result: it carries the error that
    bf16 activations accumulate over up to M x J layer applications (the same
    error the logits carry) plus one bf16 storage rounding (<= 2^-9 of the
    entry), normalised by the max of a row of Hkv x hd values.
    * Entries written by decode steps (two-term GEMM operands): measured worst
      3.9e-3 over the C3/C4/C5 snapshot runs; bar 1e-2.
    * Caches that also hold prefilled entries: the prefill GEMMs take one bf16
      plane per operand, so each layer application adds about four roundings of
      up to 2^-9 relative, and they add up like a random walk: over the 12
      layer applications of the C4 model's deepest loop that is about 1.4e-2
      for a typical row and up to about twice that for the worst of tens of
      thousands of rows. Measured worst 2.04e-2 (C4 model, loop 6); bar 3e-2.
    """
    if model.dtype == "f32":
        return 1e-4
    return 3e-2 if prefilled else 1e-2


def check_cache(ctx, seq_id, oseq, model, tol=None, masked_slots=False):
    """GPU cache of one sequence against the oracle's: positions exact, K/V within tol.

    masked_slots: the cache keeps a slot per position (dense-cache ablation); slot t
    of loop i must hold position t if the token ran loop i, else the mask -1, and
    the K/V of the unmasked slots are compared.
    """
    tol = cache_tol(model) if tol is None else tol
    worst = 0.0
    for i in range(model.max_loops):
        for j in range(model.n_layers):
            gp, gk, gv = ctx.read_cache(seq_id, i + 1, j)
            op, ok, ov = oseq.caches[i][j].view()
            if masked_slots:
                want = np.full(len(gp), -1, dtype=np.int64)
                want[np.asarray(op, dtype=np.int64)] = op
                np.testing.assert_array_equal(gp, want)
                keep = np.asarray(gp) >= 0
                gp, gk, gv = gp[keep], gk[keep], gv[keep]
            np.testing.assert_array_equal(gp, op)
            for name, g, o in (("k", gk, ok), ("v", gv, ov)):
                if not len(op):
                    continue
                g2, o2 = g.reshape(len(op), -1).astype(np.float64), o.reshape(len(op), -1).astype(np.float64)
                row = np.max(np.abs(g2 - o2), axis=1) / np.max(np.abs(o2), axis=1)
                bad = int(np.argmax(row))
                worst = max(worst, float(row[bad]))
                assert row[bad] < tol, (f"cache {name} loop {i + 1} layer {j}: entry {bad}/{len(op)} "
                                        f"(pos {op[bad]}) rel err {row[bad]:.3e}; rows over tol: "
                                        f"{np.nonzero(row >= tol)[0][:10].tolist()} gpu {g2[bad, :4]} "
                                        f"oracle {o2[bad, :4]}")
    print(f"cache of sequence {seq_id}: worst K/V row rel err {worst:.3e} (bar {tol:.0e})")
    return worst
