"""tlf_attn_decode_static: the attention entry point for callers that cannot allocate.

Some callers have no way to allocate device memory (their host application
owns the GPU's memory through its own pool, or their request path forbids a
cudaMalloc that could synchronise the device). This entry point serves them
from a fixed 4 MiB array built into the library. Its results must equal those
of tlf_attn_decode with caller scratch bit for bit and match the oracle;
successive calls on different inputs check that the array's leftover contents
from one call never leak into the next. This file is collected last so that
a failure here stops a first-failure run only after every other test has run.
"""
import numpy as np
import pytest

from oracle import tlf_oracle as O

from _attn_problem import args_for, gather_kv, make_problem, out_to_host, to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def T():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2609_15160_gb300 import build, tlf
    build.build()
    tlf.load_library()
    return tlf


def _with_caller_scratch(T, p):
    import torch
    d = to_device(p)
    a = args_for(T, p, d)
    nbytes = T.tlf_attn_decode_scratch_bytes(a)
    scratch = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    T.tlf_attn_decode(a, scratch, nbytes)
    torch.cuda.synchronize()
    assert int(d["err"][0].item()) == 0
    return out_to_host(p, d["out"]), nbytes


def _matches_oracle(p, got, tol=2e-2):
    """Every row against the oracle's attention over that row's keys (bf16 output: 2e-2)."""
    for b in range(p["n"]):
        k, v = gather_kv(p, b)
        want = O.attention(p["q"][b].astype(np.float64), k, v)
        err = np.max(np.abs(got[b] - want)) / np.max(np.abs(want))
        assert err < tol, (b, err)


def test_static_scratch_matches_caller_scratch_on_successive_calls(T):
    """Three calls in a row on different inputs, each bit-identical to the caller-scratch entry
    point (the same kernels on the same grid and plan) and within 2e-2 of the oracle. The
    third call passes no error word, so the entry point clears its own word in the array, and
    its row lengths differ from the call before, so stale plan entries, partials or merge
    tickets left in the array would change its output."""
    import torch
    problems = [
        make_problem(16, [32768] * 2 + [1, 63, 64, 65, 129, 4000] + [2048] * 8, 16, 8, 128, seed=21),
        make_problem(5, [7, 300, 1, 64, 9000], 16, 16, 64, seed=22),
        make_problem(7, [5000, 2, 129, 64, 1, 800, 31], 16, 16, 64, seed=24),
    ]
    for i, p in enumerate(problems):
        want, nbytes = _with_caller_scratch(T, p)
        assert nbytes <= 4 << 20
        d = to_device(p)
        d["out"].fill_(0x7FC0)   # garbage in the output before the call
        with_err = i < 2
        a = args_for(T, p, d) if with_err else T.attn_args(
            p["n"], p["hq"], p["hkv"], p["hd"], p["n_layers"], p["layer"], p["dtype"], p["max_pages"],
            p["n_pages"], d["q"], d["pool"], d["page_table"], d["lens"], d["out"], None)
        T.tlf_attn_decode_static(a)
        torch.cuda.synchronize()
        if with_err:
            assert int(d["err"][0].item()) == 0
        got = out_to_host(p, d["out"])
        assert np.array_equal(got, want), f"call {i}: max diff {np.max(np.abs(got - want))}"
        _matches_oracle(p, got)


def test_static_scratch_rejects_oversized_calls(T):
    # 256 rows x 16 kv heads x 4 query heads each of 128: the split-K partials alone need ~9.6 MB
    p = make_problem(256, [10] * 256, 64, 16, 128, n_layers=1, layer=0, seed=23)
    d = to_device(p)
    a = args_for(T, p, d)
    assert T.tlf_attn_decode_scratch_bytes(a) > 4 << 20
    with pytest.raises(T.TlfError, match="built-in buffer holds 4194304"):
        T.tlf_attn_decode_static(a)
