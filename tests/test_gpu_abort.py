"""The bf16 attention kernel's own abort path, driven by a planted missing load.

cover_debug_attn_fault launches the production kernel with one CTA leaving out
the K tile load of one of its KV ring entries and every bounded wait limited to
a few milliseconds. The waits that depend on that tile run out: the test checks
that the launch returns well within a second, that COVER_ERR_DEVICE_TIMEOUT is
recorded by the faulted CTA (and cleared by the read), that every row the
other CTAs own is bit-identical to a clean launch, and that the next clean
launch is bit-identical again. No wait is left unbounded, nothing traps, and
the context stays usable throughout.
"""
import time

import numpy as np
import pytest
import torch

from paper_2602_06161_gb300 import api
from paper_2602_06161_gb300 import workloads as W
from tests import _gpu as H

pytestmark = pytest.mark.gpu

LIMIT_US = 20000                      # 20 ms per wait
SITES = {10, 20, 30, 31, 40, 50, 51}  # TMA, MMA, softmax 0/1, routing, seed-score warps
N_SM = 152


def _rows_of_cta(c, B, Hq, Lq, grid, n_split_rows):
    """(b, hq, row range) the persistent grid gives CTA c in these launches: units c, c + grid, ...
    of 256 rows; n_split_rows > 0 marks a launch whose units are all split over CTA pairs."""
    n_mblk = (Lq + 255) // 256
    n_units = n_mblk * Hq * B
    owned = []
    if n_split_rows:
        u, t = c // 2, c % 2
        mblk, bh = u % n_mblk, u // n_mblk
        owned.append((bh // Hq, bh % Hq, mblk * 256 + t * 128, mblk * 256 + t * 128 + 128))
        return owned
    for u in range(c, n_units, grid):
        mblk, bh = u % n_mblk, u // n_mblk
        owned.append((bh // Hq, bh % Hq, mblk * 256, mblk * 256 + 256))
    return owned


CASES = [
    # name, (B, Hq, Hkv, Lq, Lk, q0, S), fault entry, grid, split
    ("square_two_units_first_load", (2, 32, 8, 1024, 1024, 0, 24), 0, N_SM, 0),
    ("square_two_units_mid_unit", (2, 32, 8, 1024, 1024, 0, 24), 5, N_SM, 0),
    ("square_two_units_boundary", (2, 32, 8, 1024, 1024, 0, 24), 9, N_SM, 0),
    ("square_two_units_last_load", (2, 32, 8, 1024, 1024, 0, 24), 15, N_SM, 0),
    ("square_split_units", (1, 8, 8, 1024, 1024, 0, 16), 3, 64, 1),
    ("window_split_halves", (1, 4, 2, 64, 1024, 512, 12), 2, 4, 0),
]


@pytest.mark.parametrize("name,shape,entry,grid,split", CASES, ids=[c[0] for c in CASES])
def test_planted_missing_load_aborts_cleanly(name, shape, entry, grid, split):
    B, Hq, Hkv, Lq, Lk, q0, S = shape
    inp = W.make_attn_inputs(B, Hq, Hkv, Lk, 128, S, dtype="bf16", seed=61, seed_lo=q0, seed_hi=q0 + Lq)
    dev = [H.to_dev(inp.q[:, :, q0:q0 + Lq], "bf16"), H.to_dev(inp.k_cached, "bf16"),
           H.to_dev(inp.v_cached, "bf16"), H.to_dev(inp.k_seedmask, "bf16"), H.to_dev(inp.v_seedmask, "bf16"),
           H.to_dev(inp.seed_idx, "i32")]
    # the clean launch of the same kernel: the fault entry with no planted load. A square call of
    # the production entry runs that kernel too and must give the same bits; a short window of
    # grouped-query heads runs on the packed window kernel instead, which agrees up to rounding.
    clean, clean_lse = api.cover_debug_attn_fault(*dev, q0=q0, fault_cta=-1, fault_entry=-1, limit_us=LIMIT_US)
    prod, prod_lse = api.cover_attn_fwd_prefix(*dev, q0=q0)
    torch.cuda.synchronize()
    assert api.cover_debug_status_detail() == (0, 0, 0)
    if Lq == Lk and q0 == 0:
        assert torch.equal(prod, clean) and torch.equal(prod_lse, clean_lse)
    else:
        assert (prod.float() - clean.float()).abs().max().item() <= H.TOL_BF16_MAX
        assert (prod_lse - clean_lse).abs().max().item() <= H.TOL_LSE

    out = torch.full_like(clean, float("nan"))
    lse = torch.full_like(clean_lse, float("nan"))
    t0 = time.perf_counter()
    api.cover_debug_attn_fault(*dev, q0=q0, fault_cta=0, fault_entry=entry, limit_us=LIMIT_US, out=out, lse=lse)
    code, site, block = api.cover_debug_status_detail()
    elapsed = time.perf_counter() - t0
    print(f"{name}: site {site}, block {block}, {elapsed * 1e3:.1f} ms")
    assert code == -4 and site in SITES and block == 0, (code, site, block)
    assert elapsed < 0.5
    assert api.cover_debug_status_detail() == (0, 0, 0)     # the read cleared it

    # every row that another CTA owns is exactly the clean result
    mine = torch.zeros((B, Hq, Lq), dtype=torch.bool, device="cuda")
    for b, hq, r0, r1 in _rows_of_cta(0, B, Hq, Lq, grid, split):
        mine[b, hq, r0:min(r1, Lq)] = True
    assert mine.any() and not mine.all()
    assert torch.equal(out[~mine], clean[~mine]) and torch.equal(lse[~mine], clean_lse[~mine])

    # the context is usable and the kernel leaves nothing behind: a clean launch matches again
    again, again_lse = api.cover_debug_attn_fault(*dev, q0=q0, fault_cta=-1, fault_entry=-1, limit_us=LIMIT_US)
    prod_again, prod_again_lse = api.cover_attn_fwd_prefix(*dev, q0=q0)
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    assert torch.equal(again, clean) and torch.equal(again_lse, clean_lse)
    assert torch.equal(prod_again, prod) and torch.equal(prod_again_lse, prod_lse)


def test_fault_entry_beyond_the_ctas_work_plants_nothing():
    inp = W.make_attn_inputs(1, 4, 4, 512, 128, 6, dtype="bf16", seed=62)
    dev = [H.to_dev(inp.q, "bf16"), H.to_dev(inp.k_cached, "bf16"), H.to_dev(inp.v_cached, "bf16"),
           H.to_dev(inp.k_seedmask, "bf16"), H.to_dev(inp.v_seedmask, "bf16"), H.to_dev(inp.seed_idx, "i32")]
    clean, clean_lse = api.cover_attn_fwd(*dev)
    out, lse = api.cover_debug_attn_fault(*dev, fault_cta=0, fault_entry=10 ** 6, limit_us=LIMIT_US)
    assert api.cover_debug_status_detail() == (0, 0, 0)
    assert torch.equal(out, clean) and torch.equal(lse, clean_lse)
    ref, ref_lse = H.oracle_full(inp)
    H.assert_bf16_close(out.float().cpu().numpy().astype(np.float64), ref, lse.cpu().numpy(), ref_lse)
