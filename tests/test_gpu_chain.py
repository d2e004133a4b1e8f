"""Kernels of the library launched back to back on one stream, each a programmatic dependent of
the one before: every kernel must read what the previous one wrote. The chain of one decoding
step (seed K/V gather, override swap, attention, d_in / d_out from the attention's lse, the
selection with them) runs once with no host synchronisation between the calls and once with a
synchronisation after each; every output must be bit-identical."""
import numpy as np
import pytest
import torch

from paper_2602_06161_gb300 import api
from paper_2602_06161_gb300 import workloads as W
from tests import _gpu as H

pytestmark = pytest.mark.gpu


def _inputs():
    B, Hq, Hkv, L, S, per = 2, 4, 2, 640, 24, 256
    inp = W.make_attn_inputs(B, Hq, Hkv, L, 128, S, dtype="bf16", seed=31)
    rng = np.random.default_rng(32)
    prev = W.make_attn_inputs(B, Hq, Hkv, L, 128, S, dtype="bf16", seed=33)   # the previous step's K, V
    tok = rng.integers(0, 6, size=B * per).astype(np.int32)
    masked = rng.random(B * per) < 0.4
    tok[masked] = 7
    flags = np.zeros(B * per, np.uint8)
    flags[(~masked) & (rng.random(B * per) < 0.3)] |= 2
    d = dict(q=H.to_dev(inp.q, "bf16"), k=H.to_dev(inp.k_cached, "bf16"), v=H.to_dev(inp.v_cached, "bf16"),
             kp=H.to_dev(prev.k_cached, "bf16"), vp=H.to_dev(prev.v_cached, "bf16"),
             seeds=H.to_dev(inp.seed_idx, "i32"), tok=torch.from_numpy(tok).cuda(),
             flags=torch.from_numpy(flags).cuda())
    return d, (B, Hq, Hkv, L, S, per)


def _chain(d, dims, sync):
    B, Hq, Hkv, L, S, per = dims
    k, v = d["k"].clone(), d["v"].clone()
    kc = torch.full((B, Hkv, S, 128), float("nan"), dtype=torch.bfloat16, device="cuda")
    vc = torch.full_like(kc, float("nan"))
    out = torch.full_like(d["q"], float("nan"))
    lse = torch.full((B, Hq, L), float("nan"), device="cuda")
    mws = torch.empty((api.cover_attn_mass_workspace_bytes(B, Hq, per) + 15) // 16, 4, dtype=torch.int32,
                      device="cuda")
    d_in = torch.full((B * per,), float("nan"), device="cuda")
    d_out = torch.full_like(d_in, float("nan"))
    torch.cuda.synchronize()

    def step():
        if sync:
            torch.cuda.synchronize()

    api.cover_seed_kv_gather(d["kp"], d["vp"], d["seeds"], k_cache=kc, v_cache=vc)
    step()
    api.cover_seed_kv_override(k, v, d["seeds"], kc, vc)
    step()
    api.cover_attn_fwd(d["q"], k, v, kc, vc, d["seeds"], out=out, lse=lse)
    step()
    api.cover_attn_mass_fwd(d["q"], k, lse, d["tok"], d["flags"], mask_id=7, pos0=L - per, per=per,
                            k_seedmask=kc, seed_idx=d["seeds"], workspace=mws, d_in=d_in, d_out=d_out)
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    return dict(k=k, v=v, kc=kc, vc=vc, out=out, lse=lse, d_in=d_in, d_out=d_out)


def test_back_to_back_launches_read_their_predecessors_results():
    d, dims = _inputs()
    a = _chain(d, dims, sync=False)
    b = _chain(d, dims, sync=True)
    for name in a:
        assert not torch.isnan(a[name].float()).any(), name
        assert torch.equal(a[name], b[name]), name
