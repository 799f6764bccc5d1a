"""The kernel-level recursion-wise attention (tlf_attn_decode) against the oracle's attention."""
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


CASES = [
    # (lens, hq, hkv, hd, dtype)
    ([1, 63, 64, 65, 3000, 40000], 16, 8, 128, "bf16"),
    ([2048] * 5 + [1, 700], 16, 16, 64, "bf16"),
    ([5, 129, 1000], 8, 2, 128, "bf16"),
    ([33, 64, 500], 4, 2, 32, "bf16"),
    ([1, 31, 200], 4, 4, 16, "f32"),
    ([77] * 256, 4, 2, 64, "bf16"),
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: f"hd{c[3]}-g{c[1] // c[2]}-{c[4]}-n{len(c[0])}")
def test_attention_op_matches_oracle(T, case):
    import torch
    lens, hq, hkv, hd, dtype = case
    p = make_problem(len(lens), lens, hq, hkv, hd, dtype=dtype, seed=len(lens) + hd)
    d = to_device(p)
    a = args_for(T, p, d)
    nbytes = T.tlf_attn_decode_scratch_bytes(a)
    assert nbytes > 0
    scratch = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    T.tlf_attn_decode(a, scratch, nbytes)
    torch.cuda.synchronize()
    assert int(d["err"][0].item()) == 0
    got = out_to_host(p, d["out"])
    tol = 1e-4 if dtype == "f32" else 2e-2
    for b in range(p["n"]):
        k, v = gather_kv(p, b)
        want = O.attention(p["q"][b].astype(np.float64), k, v)
        err = np.max(np.abs(got[b] - want)) / np.max(np.abs(want))
        assert err < tol, (b, err)


def test_attention_op_rejects_bad_arguments(T):
    import torch
    p = make_problem(2, [10, 20], 4, 2, 64)
    d = to_device(p)
    a = args_for(T, p, d)
    a.page_size = 32
    assert T.tlf_attn_decode_scratch_bytes(a) == 0
    with pytest.raises(T.TlfError):
        T.tlf_attn_decode(a, None, 0)
    a = args_for(T, p, d)
    with pytest.raises(T.TlfError, match="scratch"):
        T.tlf_attn_decode(a, torch.empty(16, dtype=torch.uint8, device="cuda"), 16)
