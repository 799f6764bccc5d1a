"""Device-side helpers of the kernel-level attention tests (inputs come from synth)."""
import numpy as np

from paper_2609_15160_gb300.synth import make_attn_problem as make_problem  # noqa: F401


def gather_kv(p, b):
    """K, V [len, hkv, hd] of row b, in key order."""
    ps = p["page_size"]
    L = int(p["lens"][b])
    e = np.arange(L)
    pages = p["page_table"][b, e // ps]
    k = p["pool"][pages, p["layer"], 0, :, e % ps, :]
    v = p["pool"][pages, p["layer"], 1, :, e % ps, :]
    return k, v


def to_device(p):
    import torch
    if p["dtype"] == "bf16":
        bits = (p["pool"].view(np.uint32) >> 16).astype(np.uint16).view(np.int16)
        pool = torch.from_numpy(bits).cuda()
        out = torch.zeros((p["n"], p["hq"] * p["hd"]), dtype=torch.int16, device="cuda")
    else:
        pool = torch.from_numpy(p["pool"]).cuda()
        out = torch.zeros((p["n"], p["hq"] * p["hd"]), dtype=torch.float32, device="cuda")
    return dict(q=torch.from_numpy(p["q"]).cuda(), pool=pool, page_table=torch.from_numpy(p["page_table"]).cuda(),
                lens=torch.from_numpy(p["lens"]).cuda(), out=out,
                err=torch.zeros(4, dtype=torch.int32, device="cuda"))


def out_to_host(p, out):
    a = out.cpu().numpy()
    if p["dtype"] == "bf16":
        a = (a.view(np.uint16).astype(np.uint32) << 16).view(np.float32)
    return a.reshape(p["n"], p["hq"], p["hd"])


def args_for(T, p, d):
    return T.attn_args(p["n"], p["hq"], p["hkv"], p["hd"], p["n_layers"], p["layer"], p["dtype"], p["max_pages"],
                       p["n_pages"], d["q"], d["pool"], d["page_table"], d["lens"], d["out"], d["err"])
