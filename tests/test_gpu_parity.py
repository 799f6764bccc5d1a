"""GPU path vs CPU oracle on the workload configurations and edge cases.

Every call goes through the C ABI (libtlf.so) via the ctypes binding.
"""
import dataclasses

import numpy as np
import pytest

from oracle import tlf_oracle as O
from paper_2609_15160_gb300 import synth

from _parity import DepthOracle, cache_tol, check_active_sets, check_cache, rel_err, tol_for

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tlf():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2609_15160_gb300 import build, tlf as T
    build.build()
    T.load_library()
    return T


def _greedy_run(T, wl, steps=None, gemm_impl="auto", check_caches=True, ablation="none"):
    """Prefill + greedy decode, teacher-forced from the oracle's argmax."""
    m = wl.model
    w = synth.make_weights(m)
    om = O.OracleModel.from_config(m, w)
    depth = DepthOracle(om)
    prompts = synth.make_prompts(wl)
    B = len(prompts)
    steps = wl.decode_steps if steps is None else steps
    L = max(len(p) for p in prompts) + steps + 1
    ids = list(range(100, 100 + B))
    tol = tol_for(m)
    worst = 0.0
    with T.Context(m, w, max_seqs=B, max_batch=B, max_seq_len=L, gemm_impl=gemm_impl, ablation=ablation) as ctx:
        pf_forced = [depth.forced_for(p) for p in prompts]
        glog, gloops = ctx.prefill(ids, prompts, forced=pf_forced)
        seqs = [O.OracleSequence(om) for _ in range(B)]
        nxt = np.zeros(B, dtype=np.int32)
        for b in range(B):
            olog, om_ = O.prefill_gathered(om, seqs[b], prompts[b], forced=pf_forced[b])
            np.testing.assert_array_equal(gloops[b], om_)
            np.testing.assert_array_equal(gloops[b], depth.expected(prompts[b], pf_forced[b]))
            worst = max(worst, rel_err(glog[b], olog))
            nxt[b] = int(np.argmax(olog))
        assert worst < tol, f"prefill logits rel err {worst}"
        for step in range(steps):
            f = depth.forced_for(nxt)
            glog, gl, gmar = ctx.decode_step(ids, nxt, forced=f)
            olog, oloops, omar = O.decode_step(om, seqs, nxt, forced=f)
            np.testing.assert_array_equal(gl, oloops)
            check_active_sets(ctx, gl, m.max_loops, ablation)
            e = rel_err(glog, olog)
            worst = max(worst, e)
            assert e < tol, f"step {step}: logits rel err {e}"
            free = f < 1
            np.testing.assert_allclose(gmar[free], omar[free], rtol=1e-3, atol=1e-4)
            nxt = np.argmax(olog, axis=1).astype(np.int32)
        if check_caches:
            dense = ablation == "dense_cache"  # every loop cache has a slot per token
            for b in range(B):
                for r in range(1, m.max_loops + 1):
                    assert ctx.cache_len(ids[b], r) == seqs[b].cache_len(1 if dense else r)
            check_cache(ctx, ids[0], seqs[0], m, masked_slots=dense)
    return worst, depth.n_forced


def test_c1_fp32_full_greedy_parity(tlf):
    worst, forced = _greedy_run(tlf, synth.get_config("c1"))
    print(f"c1 worst logits rel err {worst:.2e}, near-tie tokens forced {forced}")


def test_c2_bf16_full_greedy_parity(tlf):
    worst, forced = _greedy_run(tlf, synth.get_config("c2"))
    print(f"c2 worst logits rel err {worst:.2e}, near-tie tokens forced {forced}")


def test_c2_simt_gemm_path_matches_oracle(tlf):
    """The CUDA-core GEMM path on the same bf16 model (a second GPU path for the tcgen05 kernels)."""
    wl = synth.get_config("c2").with_batch(4)
    worst, _ = _greedy_run(tlf, wl, steps=8, gemm_impl="simt", check_caches=False)
    print(f"c2 simt worst {worst:.2e}")


def test_c2_unsplit_norm_path_matches_oracle(tlf, monkeypatch):
    """Every pre-norm as a kernel of its own (the tcgen05 path without the split norm)."""
    monkeypatch.setenv("TLF_NO_SPLIT_NORM", "1")
    worst, _ = _greedy_run(tlf, synth.get_config("c2"), steps=16)
    print(f"c2 unsplit-norm worst {worst:.2e}")


def test_one_plane_operand_path_matches_oracle(tlf, monkeypatch):
    """The tcgen05 path with single bf16 GEMM operands (no lo planes)."""
    monkeypatch.setenv("TLF_NO_OPERAND_LO", "1")
    worst, _ = _greedy_run(tlf, synth.get_config("c2"), steps=16)
    print(f"c2 one-plane worst {worst:.2e}")


def _snapshot_run(T, wl, lengths, steps, sampled, seed=7, distinct=2, ablation="none", host_values="all"):
    """Sequences restored from synthetic cache snapshots, then decode steps of random tokens.

    Loop counts and active sets are checked for every token (against the
    oracle's depth table, or the workload's forced depth); logits and caches
    for the sampled sequences. host_values="sampled" uploads host K/V values
    only for the sampled sequences and lets the device fill the others (their
    values do not matter: sequences are independent, and only loop counts,
    active sets and cache lengths are checked for them), which keeps wide
    batches within host memory.
    """
    m = wl.model
    w = synth.make_weights(m)
    om = O.OracleModel.from_config(m, w)
    depth = DepthOracle(om)
    B = len(lengths)
    fixed = wl.forced_loops
    if host_values == "sampled":
        distinct = B  # one snapshot per sequence, so no unsampled sequence shares a sampled one's values
    snaps = {}
    for b in range(B):
        L = int(lengths[b])
        key = (L, b % distinct)
        if key not in snaps:
            sd = seed + 31 * key[1] + L
            depths = None if fixed is None else np.full(L, fixed, np.int32)
            make = synth.make_cache_snapshot if (host_values == "all" or b in sampled) else synth.make_cache_positions
            snaps[key] = make(m, L, sd, depths=depths)
    snap_of = [snaps[(int(lengths[b]), b % distinct)] for b in range(B)]
    pages = sum(sum((len(p) + 63) // 64 + 1 for p in snap["positions"]) for snap in snap_of) + \
        B * m.max_loops * (steps // 64 + 2)
    if ablation == "dense_cache":  # every loop cache holds a slot per position
        pages = B * m.max_loops * ((int(max(lengths)) + steps) // 64 + 2)
    ids = list(range(1000, 1000 + B))
    tokens = synth.make_decode_tokens(wl, steps=steps, batch=B)
    tol = tol_for(m)
    worst = 0.0
    with T.Context(m, w, max_seqs=B, max_batch=B, max_seq_len=int(max(lengths)) + steps + 1,
                   kv_pool_pages=pages, ablation=ablation) as ctx:
        for b in range(B):
            ctx.load_cache(ids[b], snap_of[b])
        oseqs = {b: O.load_snapshot(om, snap_of[b], cache_dtype=np.float32) for b in sampled}
        all_loops = []
        for step in range(steps):
            f = depth.forced_for(tokens[step]) if fixed is None else np.full(B, fixed, np.int32)
            glog, gl, _ = ctx.decode_step(ids, tokens[step], forced=f)
            np.testing.assert_array_equal(gl, depth.expected(tokens[step], f))
            check_active_sets(ctx, gl, m.max_loops, ablation)
            all_loops.append(gl.copy())
            for b in sampled:
                olog, oml, _ = O.decode_token(om, oseqs[b], int(tokens[step][b]), forced=int(f[b]))
                assert oml == gl[b]
                e = rel_err(glog[b], olog)
                worst = max(worst, e)
                assert e < tol, f"step {step} seq {b}: rel err {e}"
        all_loops = np.array(all_loops)
        dense = ablation == "dense_cache"
        for b in range(B):
            snap = snap_of[b]
            for r in range(1, m.max_loops + 1):
                if dense:
                    want = len(snap["positions"][0]) + steps
                else:
                    want = len(snap["positions"][r - 1]) + int((all_loops[:, b] >= r).sum())
                assert ctx.cache_len(ids[b], r) == want
        for b in sampled:  # restored entries are exact; every other entry was written by a decode step
            check_cache(ctx, ids[b], oseqs[b], m, tol=cache_tol(m, prefilled=False), masked_slots=dense)
    return worst, depth.n_forced


def test_c3_full_size_sampled_parity(tlf):
    wl = synth.get_config("c3")
    lengths = np.full(wl.batch, wl.prompt_len[0])
    worst, forced = _snapshot_run(tlf, wl, lengths, steps=4, sampled=[0, 37])
    print(f"c3 worst {worst:.2e} forced {forced}")


def test_two_term_operands_keep_deep_models_precise(tlf):
    """C3 (8 loops x 4 layers) at 16 tokens: with hi + lo bf16 GEMM operands the logits stay
    within 5e-3 of the float64 oracle, a quarter of the 2e-2 bound (one bf16 plane: about 1.9e-2)."""
    wl = synth.get_config("c3")
    lengths = np.full(16, wl.prompt_len[0])
    worst, _ = _snapshot_run(tlf, wl.with_batch(16), lengths, steps=3, sampled=[0, 5])
    assert worst < 5e-3, worst


def test_c4_full_size_sampled_parity(tlf):
    wl = synth.get_config("c4")
    lengths = np.full(wl.batch, wl.prompt_len[0])
    worst, forced = _snapshot_run(tlf, wl, lengths, steps=3, sampled=[0, 9])
    print(f"c4 worst {worst:.2e} forced {forced}")


def _c5_run(T, name, batch, steps=3):
    """The ragged C5 sweep workload at one batch size: every token's loop count and active sets,
    the logits and caches of the longest and the shortest sequence."""
    wl = synth.get_config(name).with_batch(batch)
    lengths = np.array([len(p) for p in synth.make_prompts(wl)])
    sampled = sorted({int(np.argmax(lengths)), int(np.argmin(lengths))})
    worst, forced = _snapshot_run(T, wl, lengths, steps=steps, sampled=sampled, host_values="sampled")
    print(f"{name} B {batch} worst logits rel err {worst:.2e} near-tie tokens forced {forced}")
    return worst


def test_c5_ragged_sampled_parity(tlf):
    _c5_run(tlf, "c5", 32)


def test_c5_forced8_sampled_parity(tlf):
    """The fixed-depth baseline run of the sweep: every past and new token at 8 loops."""
    _c5_run(tlf, "c5f", 32)


@pytest.mark.parametrize("name", ["c5", "c5f"])
@pytest.mark.parametrize("batch", [128, 256])
def test_c5_wide_batch_sampled_parity(tlf, name, batch):
    """C5 at the sweep's wide batches (token tiles of 128 and 256 in the GEMMs, two-term operands):
    the 8-loop x 4-layer model stays within 5e-3 of the oracle, a quarter of the 2e-2 bound."""
    assert _c5_run(tlf, name, batch) < 5e-3


def _prefill_full_size(T, name, lens, chunk, steps=3, seed=29):
    """Prompts of the workload's model through the batched prefill, then decode steps, against the oracle.

    Checks every prompt token's loop count, the logits after each prompt, every
    (loop, layer) cache entry (positions exact, K/V within the cache tolerance)
    and then the logits of a few decode steps that read those caches.
    """
    m = synth.get_config(name).model
    w = synth.make_weights(m)
    om = O.OracleModel.from_config(m, w)
    depth = DepthOracle(om)
    rng = np.random.default_rng(seed)
    prompts = [rng.integers(0, m.vocab, size=n).astype(np.int32) for n in lens]
    B = len(prompts)
    ids = [40 + b for b in range(B)]
    tol = tol_for(m)
    worst_pf = worst_dec = 0.0
    with T.Context(m, w, max_seqs=B, max_batch=B, max_seq_len=max(lens) + steps + 1, prefill_chunk=chunk) as ctx:
        pf = [depth.forced_for(p) for p in prompts]
        glog, gl = ctx.prefill(ids, prompts, forced=pf)
        seqs = [O.OracleSequence(om) for _ in range(B)]
        for b in range(B):
            olog, oml = O.prefill_gathered(om, seqs[b], prompts[b], forced=pf[b])
            np.testing.assert_array_equal(gl[b], oml)
            np.testing.assert_array_equal(gl[b], depth.expected(prompts[b], pf[b]))
            e = rel_err(glog[b], olog)
            worst_pf = max(worst_pf, e)
            assert e < tol, f"prompt {b}: last-token logits rel err {e}"
            for r in range(1, m.max_loops + 1):
                assert ctx.cache_len(ids[b], r) == seqs[b].cache_len(r)
            check_cache(ctx, ids[b], seqs[b], m)
        for step in range(steps):
            toks = rng.integers(0, m.vocab, size=B).astype(np.int32)
            f = depth.forced_for(toks)
            glog, gm, _ = ctx.decode_step(ids, toks, forced=f)
            olog, om2, _ = O.decode_step(om, seqs, toks, forced=f)
            np.testing.assert_array_equal(gm, om2)
            check_active_sets(ctx, gm, m.max_loops)
            e = rel_err(glog, olog)
            worst_dec = max(worst_dec, e)
            assert e < tol, f"decode step {step}: logits rel err {e}"
    print(f"{name} prefill {lens} chunk {chunk}: worst prefill logits {worst_pf:.2e}, decode {worst_dec:.2e}, "
          f"near-tie tokens forced {depth.n_forced}")
    return worst_pf, worst_dec


def test_c4_model_prefill_two_chunks(tlf):
    """C4 model (hd 128, GQA 2): a 3000-token prompt over two 2048-token chunks, the second shared with a
    700-token prompt; the windowed GEMM epilogues and the chunk-to-chunk cache slots of App. B."""
    _prefill_full_size(tlf, "c4", [3000, 700], chunk=2048)


def test_c3_model_prefill_one_chunk(tlf):
    """C3 model (8 loops x 4 layers): two prompts of 2048 and 1500 tokens in one chunk."""
    _prefill_full_size(tlf, "c3", [2048, 1500], chunk=8192)


# ----------------------------------------------------------------------------
# edge cases on small models
# ----------------------------------------------------------------------------

def _small(dtype="bf16", **kw):
    base = dict(vocab=300, d_model=128, n_heads=4, n_kv_heads=2, head_dim=64, n_layers=2, ffn_hidden=160,
                max_loops=4, dtype=dtype, depth_probs=(0.25, 0.25, 0.25, 0.25))
    if dtype == "f32":
        base["depth_probs"] = None
    base.update(kw)
    return synth.ModelConfig(**base)


def _prefill_decode_compare(T, m, prompt_lens, steps, forced_mode=None, seed=0, gemm_impl="auto", ablation="none"):
    w = synth.make_weights(m)
    om = O.OracleModel.from_config(m, w)
    depth = DepthOracle(om)
    rng = np.random.default_rng(seed)
    prompts = [rng.integers(0, m.vocab, size=n).astype(np.int32) for n in prompt_lens]
    B = len(prompts)
    ids = [7 * b + 3 for b in range(B)]
    tol = tol_for(m)

    def forced_of(toks):
        if forced_mode is None:
            return depth.forced_for(toks)
        if forced_mode == "random":
            return rng.integers(1, m.max_loops + 1, size=len(toks)).astype(np.int32)
        return np.full(len(toks), forced_mode, dtype=np.int32)

    with T.Context(m, w, max_seqs=B + 1, max_batch=B, max_seq_len=max(prompt_lens) + steps + 2,
                   gemm_impl=gemm_impl, ablation=ablation) as ctx:
        pf = [forced_of(p) for p in prompts]
        glog, gl = ctx.prefill(ids, prompts, forced=pf)
        seqs = [O.OracleSequence(om) for _ in range(B)]
        for b in range(B):
            olog, oml = O.prefill_gathered(om, seqs[b], prompts[b], forced=pf[b])
            np.testing.assert_array_equal(gl[b], oml)
            assert rel_err(glog[b], olog) < tol
        for s in range(steps):
            toks = rng.integers(0, m.vocab, size=B).astype(np.int32)
            f = forced_of(toks)
            glog, gm, _ = ctx.decode_step(ids, toks, forced=f)
            olog, om2, _ = O.decode_step(om, seqs, toks, forced=f)
            np.testing.assert_array_equal(gm, om2)
            check_active_sets(ctx, gm, m.max_loops, ablation)
            assert rel_err(glog, olog) < tol
        for b in range(B):
            check_cache(ctx, ids[b], seqs[b], m, masked_slots=ablation == "dense_cache")
        live, free, total = ctx.stats()
        for i in ids:
            ctx.release(i)
        assert ctx.stats() == (0, total, total)


@pytest.mark.parametrize("lens", [[1], [63, 64, 65], [128, 1, 129]])
def test_page_boundaries_and_ragged_batches(tlf, lens):
    _prefill_decode_compare(tlf, _small(), lens, steps=3)


@pytest.mark.parametrize("gqa", [(4, 4), (4, 2), (8, 2)])
def test_gqa_ratios(tlf, gqa):
    _prefill_decode_compare(tlf, _small(n_heads=gqa[0], n_kv_heads=gqa[1], d_model=256), [40, 70], steps=2)


@pytest.mark.parametrize("hd", [32, 128])
def test_head_dims(tlf, hd):
    _prefill_decode_compare(tlf, _small(head_dim=hd, n_heads=4, n_kv_heads=2, d_model=256), [66, 3], steps=2)


@pytest.mark.parametrize("hd,gqa", [(64, (4, 4)), (128, (8, 2))])
def test_thread_staged_prefill_attention_path(tlf, monkeypatch, hd, gqa):
    """The prefill attention that stages and re-lays out every K/V page with its threads
    (TLF_PF_ATTN_V1=1), the comparison path of the tensor-map kernel, on multi-page prompts."""
    monkeypatch.setenv("TLF_PF_ATTN_V1", "1")
    m = _small(head_dim=hd, n_heads=gqa[0], n_kv_heads=gqa[1], d_model=256)
    _prefill_decode_compare(tlf, m, [300, 65, 1], steps=2)


def test_every_token_exits_after_one_loop(tlf):
    """Deeper loops have no active token (device-side counts are zero)."""
    _prefill_decode_compare(tlf, _small(), [30, 65], steps=3, forced_mode=1)


def test_fixed_depth_mode(tlf):
    """Every token forced to M loops: the fixed-depth looped transformer."""
    _prefill_decode_compare(tlf, _small(), [30, 65], steps=3, forced_mode=4)


def test_random_forced_depths(tlf):
    _prefill_decode_compare(tlf, _small(max_loops=6, depth_probs=None), [100, 7, 64], steps=4, forced_mode="random")


def test_survival_exit_rule(tlf):
    _prefill_decode_compare(tlf, _small(exit_rule="survival", depth_probs=None), [50, 20], steps=3)


def test_fp32_small_model(tlf):
    _prefill_decode_compare(tlf, _small(dtype="f32", head_dim=32, n_heads=4, n_kv_heads=2), [70, 5], steps=3)


def test_wide_batch(tlf):
    """A batch larger than one MMA N tile (n > 128 tokens)."""
    m = _small(vocab=500, max_loops=3, depth_probs=(0.3, 0.3, 0.4))
    _prefill_decode_compare(tlf, m, [3 + (b % 5) for b in range(160)], steps=2)


@pytest.mark.parametrize("split", [True, False])
def test_profile_counters(tlf, monkeypatch, split):
    if not split:
        monkeypatch.setenv("TLF_NO_SPLIT_NORM", "1")
    m = _small()
    w = synth.make_weights(m)
    with tlf.Context(m, w, max_seqs=2, max_batch=2, max_seq_len=200) as ctx:
        ctx.prefill([1, 2], [np.arange(100, dtype=np.int32) % m.vocab, np.arange(10, dtype=np.int32)], logits=False)
        ctx.set_profiling(True)
        _, loops, _ = ctx.decode_step([1, 2], [5, 6])
        ms, by, nl = ctx.last_step_profile()
        # router, plan; per (loop, layer): QKV (+RoPE/append), attention, O, gate/up (+SwiGLU), down and
        # the two pre-norms, of which the split path launches only the step's first; final norm, LM head
        per = 5 if split else 7
        assert ms > 0 and nl == 2 + m.max_loops * m.n_layers * per + (1 if split else 0) + 1 + 1
        want = sum((ctx.cache_len(i, r)) * m.n_layers * 2 * m.n_kv_heads * m.head_dim * 2
                   for i, lp in zip([1, 2], loops) for r in range(1, lp + 1))
        assert abs(by - want) < 1e-6 * want


@pytest.mark.parametrize("lens", [[600, 5, 257], [300] * 3 + [1] * 70])
def test_chunked_batched_prefill(tlf, lens):
    """Prompts spanning several 256-token prefill chunks (and more sequences than one chunk holds)."""
    m = _small(vocab=400, max_loops=3, depth_probs=(0.3, 0.3, 0.4))
    w = synth.make_weights(m)
    om = O.OracleModel.from_config(m, w)
    depth = DepthOracle(om)
    rng = np.random.default_rng(17)
    prompts = [rng.integers(0, m.vocab, size=n).astype(np.int32) for n in lens]
    ids = list(range(50, 50 + len(prompts)))
    with tlf.Context(m, w, max_seqs=len(prompts), max_batch=min(64, len(prompts)), max_seq_len=700,
                     prefill_chunk=256) as ctx:
        pf = [depth.forced_for(p) for p in prompts]
        glog, gl = ctx.prefill(ids, prompts, forced=pf)
        for b in (0, 1, 2, len(prompts) - 1):
            seq = O.OracleSequence(om)
            olog, oml = O.prefill_gathered(om, seq, prompts[b], forced=pf[b])
            np.testing.assert_array_equal(gl[b], oml)
            assert rel_err(glog[b], olog) < tol_for(m)
            check_cache(ctx, ids[b], seq, m)
        live, free, total = ctx.stats()
        used = sum(sum((ctx.cache_len(i, r) + 63) // 64 for r in range(1, m.max_loops + 1)) for i in ids)
        assert total - free == used  # the worst-case reservation was trimmed


def test_device_filled_restore(tlf):
    """tlf_load_cache without values: lengths and positions as given, values on the 1/64 grid in [-2, 2)."""
    m = _small()
    w = synth.make_weights(m)
    snap = synth.make_cache_positions(m, 300, seed=5)
    with tlf.Context(m, w, max_seqs=1, max_batch=1, max_seq_len=400) as ctx:
        ctx.load_cache(9, snap)
        for r in range(1, m.max_loops + 1):
            assert ctx.cache_len(9, r) == len(snap["positions"][r - 1])
            p, k, v = ctx.read_cache(9, r, m.n_layers - 1)
            np.testing.assert_array_equal(p, snap["positions"][r - 1])
            for a in (k, v):
                if a.size:
                    assert np.all(a * 64 == np.round(a * 64)) and a.min() >= -2 and a.max() < 2 and a.std() > 0.5
        lg, loops, _ = ctx.decode_step([9], [3])
        assert np.all(np.isfinite(lg))


def test_decode_step_is_deterministic(tlf):
    """Two contexts fed the same inputs produce bitwise identical logits and caches.

    Split-K partial sums are reduced in a fixed order inside each thread-block
    cluster and every residual element has a single writer, so no floating-point
    sum depends on scheduling.
    """
    m = _small(n_layers=2, max_loops=3, depth_probs=(0.3, 0.3, 0.4), d_model=256, n_heads=4, n_kv_heads=2)
    w = synth.make_weights(m)
    rng = np.random.default_rng(3)
    prompts = [rng.integers(0, m.vocab, size=n).astype(np.int32) for n in (100, 37, 64)]
    steps = [rng.integers(0, m.vocab, size=3).astype(np.int32) for _ in range(4)]
    outs = []
    for _ in range(2):
        with tlf.Context(m, w, max_seqs=3, max_batch=3, max_seq_len=200) as ctx:
            lg, _ = ctx.prefill([1, 2, 3], prompts)
            res = [lg]
            for t in steps:
                res.append(ctx.decode_step([1, 2, 3], t)[0])
            res.append(ctx.read_cache(1, 2, 1)[1])
            outs.append(res)
    for a, b in zip(*outs):
        np.testing.assert_array_equal(a, b)


# Launch mechanics only (no arithmetic changes): the direct-launch and plain stream-order paths
# must reproduce the graph-replayed, programmatic-dependent-launch step bit for bit.
_LAUNCH_RUN = """
import sys
import numpy as np
sys.path.insert(0, {root!r})
from paper_2609_15160_gb300 import synth, tlf as T
m = synth.ModelConfig(vocab=300, d_model=256, n_heads=4, n_kv_heads=2, head_dim=64, n_layers=2, ffn_hidden=320,
                      max_loops=3, dtype="bf16", depth_probs=(0.3, 0.3, 0.4))
w = synth.make_weights(m)
rng = np.random.default_rng(5)
prompts = [rng.integers(0, m.vocab, size=n).astype(np.int32) for n in (90, 33, 64)]
steps = [rng.integers(0, m.vocab, size=3).astype(np.int32) for _ in range(4)]
out = []
with T.Context(m, w, max_seqs=3, max_batch=3, max_seq_len=200) as ctx:
    lg, _ = ctx.prefill([1, 2, 3], prompts)
    out.append(lg)
    for t in steps:
        out.append(ctx.decode_step([1, 2, 3], t)[0])
np.save({path!r}, np.stack(out[1:]))
"""


def _launch_run(tmp_path, name, env):
    import os
    import subprocess
    import sys

    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    path = str(tmp_path / f"{name}.npy")
    r = subprocess.run([sys.executable, "-c", _LAUNCH_RUN.format(root=root, path=path)], capture_output=True,
                       text=True, env=dict(os.environ, **env), timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    return np.load(path)


def test_launch_paths_are_bitwise_identical(tlf, tmp_path):
    """Graph replay with programmatic dependent launch, direct launches (TLF_NO_GRAPH=1) and plain
    stream order (TLF_NO_PDL=1, read when the library loads) give identical decode logits."""
    base = _launch_run(tmp_path, "base", {})
    np.testing.assert_array_equal(_launch_run(tmp_path, "nograph", {"TLF_NO_GRAPH": "1"}), base)
    np.testing.assert_array_equal(_launch_run(tmp_path, "nopdl", {"TLF_NO_PDL": "1"}), base)


# ----------------------------------------------------------------------------
# ablations: the same logits and loop counts as the method, different work
# ----------------------------------------------------------------------------

def test_no_gather_ablation_c2_greedy(tlf):
    """Without the gather (every loop computes all rows, exited rows masked) the results are the method's."""
    worst, forced = _greedy_run(tlf, synth.get_config("c2"), steps=24, ablation="no_gather")
    print(f"c2 no-gather worst {worst:.2e} forced {forced}")


@pytest.mark.parametrize("gemm_impl", ["auto", "simt"])
@pytest.mark.parametrize("lens", [[1, 64, 65], [130, 2, 70, 64]])
def test_no_gather_ablation_edges(tlf, lens, gemm_impl):
    """Rows that exit with empty deeper caches (no keys at all) and page boundaries."""
    _prefill_decode_compare(tlf, _small(), lens, steps=4, gemm_impl=gemm_impl, ablation="no_gather")


def test_no_gather_ablation_c5_ragged(tlf):
    wl = synth.get_config("c5")
    lengths = np.array([len(p) for p in synth.make_prompts(wl)])
    worst, forced = _snapshot_run(tlf, wl, lengths, steps=2, sampled=[int(np.argmax(lengths)), int(np.argmin(lengths))],
                                  distinct=1, ablation="no_gather")
    print(f"c5 no-gather worst {worst:.2e} forced {forced}")


def test_dense_cache_ablation_c2_greedy(tlf):
    """Full-length caches read under the mask mu^(r) give the method's results (prefill position by position)."""
    wl = synth.get_config("c2").with_batch(4)
    worst, forced = _greedy_run(tlf, wl, steps=12, ablation="dense_cache")
    print(f"c2 dense-cache worst {worst:.2e} forced {forced}")


@pytest.mark.parametrize("lens", [[1, 64, 65], [130, 2, 70, 64]])
def test_dense_cache_ablation_edges(tlf, lens):
    _prefill_decode_compare(tlf, _small(), lens, steps=4, ablation="dense_cache")


def test_dense_cache_ablation_c3_snapshot(tlf):
    wl = synth.get_config("c3")
    lengths = np.full(16, wl.prompt_len[0])
    worst, forced = _snapshot_run(tlf, wl.with_batch(16), lengths, steps=3, sampled=[0, 5], ablation="dense_cache")
    print(f"c3 dense-cache worst {worst:.2e} forced {forced}")


# ----------------------------------------------------------------------------
# time/step AdaLN conditioning (Sec. 3.1, App. A)
# ----------------------------------------------------------------------------

def test_conditioning_c2c_greedy(tlf):
    """Per-token (depth, loop) modulation applied in the norms and residual gates, prefill and decode."""
    worst, forced = _greedy_run(tlf, synth.get_config("c2c"), steps=24)
    print(f"c2c worst {worst:.2e} forced {forced}")


def test_conditioning_c3c_full_size_sampled(tlf):
    wl = synth.get_config("c3c")
    lengths = np.full(wl.batch, wl.prompt_len[0])
    worst, forced = _snapshot_run(tlf, wl, lengths, steps=3, sampled=[0, 41])
    print(f"c3c worst {worst:.2e} forced {forced}")


@pytest.mark.parametrize("dtype,gemm_impl", [("bf16", "auto"), ("bf16", "simt"), ("f32", "auto")])
def test_conditioning_small_models(tlf, dtype, gemm_impl):
    _prefill_decode_compare(tlf, _small(dtype, conditioning=True), [70, 1, 130], steps=4, gemm_impl=gemm_impl)


def test_conditioning_with_no_gather(tlf):
    _prefill_decode_compare(tlf, _small(conditioning=True), [65, 3, 64], steps=3, ablation="no_gather")


# ----------------------------------------------------------------------------
# the two-layer MLP router (Sec. 3.2) and the survival rule at several thresholds (Eq. 4)
# ----------------------------------------------------------------------------

@pytest.mark.parametrize("dtype,gemm_impl,rule", [("bf16", "auto", "argmax"), ("bf16", "simt", "survival"),
                                                  ("f32", "auto", "argmax")])
def test_mlp_router_small_models(tlf, dtype, gemm_impl, rule):
    m = _small(dtype, router_hidden=64, exit_rule=rule)
    _prefill_decode_compare(tlf, m, [70, 1, 130], steps=4, gemm_impl=gemm_impl)


def test_mlp_router_c3_shapes(tlf):
    """C3 model with a 256-wide MLP router: every loop count and active set, sampled logits and caches."""
    wl = synth.get_config("c3")
    wl = dataclasses.replace(wl, model=dataclasses.replace(wl.model, router_hidden=256))
    lengths = np.full(wl.batch, wl.prompt_len[0])
    worst, forced = _snapshot_run(tlf, wl, lengths, steps=3, sampled=[0, 21])
    print(f"c3 mlp router worst {worst:.2e} forced {forced}")


@pytest.mark.parametrize("threshold", [0.2, 0.8])
def test_survival_thresholds_c2(tlf, threshold):
    wl = synth.get_config("c2").with_batch(4)
    wl = dataclasses.replace(wl, model=dataclasses.replace(wl.model, exit_rule="survival", threshold=threshold))
    worst, forced = _greedy_run(tlf, wl, steps=8)
    print(f"c2 survival {threshold} worst {worst:.2e} forced {forced}")
