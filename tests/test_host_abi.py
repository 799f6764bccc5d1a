"""CPU tests of the C ABI: the library loads, exports every declared symbol,
validates configurations, and a host-only context (no GPU work at all)
reports every error path while leaving its state unchanged."""
import os
import re

import ctypes as C

import numpy as np
import pytest

from paper_2609_15160_gb300 import build, synth, tlf

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return tlf.load_library()


def _declared_symbols():
    src = open(os.path.join(ROOT, "include", "tlf.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(tlf_[a-z_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared_symbols()
    for need in ("tlf_create", "tlf_prefill", "tlf_decode_step", "tlf_release", "tlf_destroy", "tlf_last_error"):
        assert need in names


def test_library_exports_every_declared_symbol(lib):
    for name in _declared_symbols():
        assert hasattr(lib, name), name
        assert name in tlf._SIGS, f"binding lacks {name}"


def _cfg(**kw):
    m = synth.get_config("c2").model
    c = tlf.make_config(m, max_seqs=4, max_batch=4, max_seq_len=256, host_only=True)
    for k, v in kw.items():
        setattr(c, k, v)
    return c


@pytest.mark.parametrize("field,value", [
    ("d_model", 100), ("n_kv_heads", 3), ("head_dim", 48), ("max_loops", 0), ("max_loops", 17),
    ("max_batch", 0), ("max_batch", 300), ("page_size", 32), ("dtype", 7), ("ffn_hidden", 1000),
    ("exit_rule", 5), ("norm_eps", 0.0), ("max_seqs", 2), ("ablation", 9), ("conditioning", 2), ("router_hidden", 12), ("router_hidden", 9000), ("reserved", 1),
])
def test_validate_config_rejects(lib, field, value):
    rc, msg = tlf.tlf_validate_config(_cfg(**{field: value}))
    assert rc == tlf.CODES["INVALID_ARG"] and msg and msg != "ok"


def test_config_struct_matches_the_header(lib):
    """The ctypes mirror of tlf_config has the C layout: int64 pool size at offset 80, then the ablation."""
    assert tlf.TlfConfig.kv_pool_pages.offset == 80 and tlf.TlfConfig.ablation.offset == 88
    assert tlf.TlfConfig.router_hidden.offset == 96 and C.sizeof(tlf.TlfConfig) == 104
    for name in ("none", "no_gather"):
        rc, msg = tlf.tlf_validate_config(_cfg(ablation=tlf.ABLATION[name]))
        assert rc == 0, msg


def test_validate_config_accepts_all_workloads(lib):
    for name, wl in synth.CONFIGS.items():
        c = tlf.make_config(wl.model, max_seqs=max(wl.batch, 256), max_batch=min(256, max(wl.batch, 1)),
                            max_seq_len=wl.prompt_len[1] + wl.decode_steps)
        rc, msg = tlf.tlf_validate_config(c)
        assert rc == 0, (name, msg)


def test_page_bytes(lib):
    m = synth.get_config("c4").model
    c = tlf.make_config(m, 16, 16, 40000)
    assert tlf.tlf_page_bytes(c) == m.n_layers * 2 * m.n_kv_heads * 64 * m.head_dim * 2
    bad = tlf.make_config(m, 16, 16, 40000)
    bad.page_size = 48
    assert tlf.tlf_page_bytes(bad) == 0


def _snapshot(m, L, seed):
    return synth.make_cache_snapshot(m, L, seed)


def test_host_only_error_paths_leave_state_unchanged(lib):
    m = synth.tiny_config(vocab=64, d_model=64, n_heads=2, n_kv_heads=1, head_dim=32, n_layers=1, ffn_hidden=64,
                          max_loops=3, dtype="bf16")
    ctx = tlf.Context(m, None, max_seqs=3, max_batch=2, max_seq_len=130, kv_pool_pages=9, host_only=True)
    try:
        assert ctx.stats() == (0, 9, 9)
        # unknown sequence
        with pytest.raises(tlf.TlfError) as e:
            ctx.decode_step([5], [1])
        assert e.value.name == "UNKNOWN_SEQ"
        # a restored sequence of 100 tokens: pages ceil(100/64) + ...
        snap = _snapshot(m, 100, 1)
        ctx.load_cache(5, snap)
        used = sum((len(p) + 63) // 64 for p in snap["positions"])
        assert ctx.stats() == (1, 9 - used, 9)
        for r in range(1, 4):
            assert ctx.cache_len(5, r) == len(snap["positions"][r - 1])
        with pytest.raises(tlf.TlfError) as e:
            ctx.load_cache(5, snap)
        assert e.value.name == "DUPLICATE_SEQ"
        # a decode step is validated and checked for pages, then refused: no GPU
        with pytest.raises(tlf.TlfError) as e:
            ctx.decode_step([5], [1])
        assert e.value.name == "NO_DEVICE"
        assert ctx.stats() == (1, 9 - used, 9)
        for bad, name in [(([5, 5], [1, 2]), "INVALID_ARG"), (([5], [64]), "INVALID_ARG"),
                          (([5, 6, 7], [1, 2, 3]), "CAPACITY")]:
            with pytest.raises(tlf.TlfError) as e:
                ctx.decode_step(*bad)
            assert e.value.name == name
        with pytest.raises(tlf.TlfError) as e:
            ctx.decode_step([5], [1], forced=[4])
        assert e.value.name == "INVALID_ARG"
        # a second long sequence exhausts the pool
        snap2 = _snapshot(m, 128, 2)
        need2 = sum((len(p) + 63) // 64 for p in snap2["positions"])
        if need2 > 9 - used:
            with pytest.raises(tlf.TlfError) as e:
                ctx.load_cache(6, snap2)
            assert e.value.name == "OUT_OF_PAGES"
            assert ctx.stats() == (1, 9 - used, 9)
        # sequence too long: a 129-token snapshot plus one step exceeds max_seq_len=130? no: exactly 130 is fine
        ctx.release(5)
        assert ctx.stats() == (0, 9, 9)
        snap3 = _snapshot(m, 129, 3)
        snap3["positions"] = [snap3["positions"][0], np.array([], np.int32), np.array([], np.int32)]
        snap3["k"] = [snap3["k"][0], snap3["k"][1][:0], snap3["k"][2][:0]]
        snap3["v"] = [snap3["v"][0], snap3["v"][1][:0], snap3["v"][2][:0]]
        ctx.load_cache(7, snap3)
        with pytest.raises(tlf.TlfError) as e:  # 129 + 1 = 130 fits; pages do not (3 for loop 1, 1 each deeper)
            ctx.decode_step([7], [1])
        assert e.value.name in ("NO_DEVICE", "OUT_OF_PAGES")
        with pytest.raises(tlf.TlfError) as e:
            ctx.release(99)
        assert e.value.name == "UNKNOWN_SEQ"
    finally:
        ctx.close()


def test_load_cache_rejects_non_nested_snapshots(lib):
    m = synth.tiny_config(vocab=64, d_model=64, n_heads=2, n_kv_heads=1, head_dim=32, n_layers=1, ffn_hidden=64,
                          max_loops=2, dtype="f32")
    ctx = tlf.Context(m, None, max_seqs=2, max_batch=1, max_seq_len=64, host_only=True)
    try:
        snap = _snapshot(m, 10, 4)
        snap["positions"][1] = np.array([0, 11], dtype=np.int32)[: len(snap["positions"][1])]
        if len(snap["positions"][1]) == 2:
            with pytest.raises(tlf.TlfError) as e:
                ctx.load_cache(1, snap)
            assert e.value.name == "INVALID_ARG"
        bad = _snapshot(m, 10, 5)
        bad["positions"][0] = bad["positions"][0][::-1].copy()
        with pytest.raises(tlf.TlfError) as e:
            ctx.load_cache(2, bad)
        assert e.value.name == "INVALID_ARG"
        assert ctx.stats()[0] == 0
    finally:
        ctx.close()


def test_binding_raises_without_library(tmp_path):
    with pytest.raises(RuntimeError, match="no fallback"):
        tlf.load_library(str(tmp_path / "missing.so"))
