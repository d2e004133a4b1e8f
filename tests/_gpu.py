"""Helpers shared by the GPU parity tests: move generator outputs to the device,
run the kernels through the binding, and evaluate the oracle on sub-problems."""
import numpy as np
import torch

import oracle
from paper_2602_06161_gb300 import api
from paper_2602_06161_gb300 import workloads as W

# tolerances: fp32 path max |d| <= 1e-5; bf16 out max |d| <= 1e-2 and mean |d| <= 1e-3; lse <= 1e-3
TOL_F32 = 1e-5
TOL_BF16_MAX = 1e-2
TOL_BF16_MEAN = 1e-3
TOL_LSE = 1e-3


def to_dev(a: np.ndarray, dtype: str):
    if dtype == "bf16":
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.bfloat16)
    if dtype == "f32":
        return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()
    if dtype == "i32":
        return torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).cuda()
    raise ValueError(dtype)


def run_attn(inp: W.AttnInputs, *, seeds_override=None):
    dt = inp.dtype
    seeds = inp.seed_idx if seeds_override is None else seeds_override
    args = [to_dev(inp.q, dt), to_dev(inp.k_cached, dt), to_dev(inp.v_cached, dt)]
    if inp.S > 0:
        args += [to_dev(inp.k_seedmask, dt), to_dev(inp.v_seedmask, dt), to_dev(seeds, "i32")]
    else:
        args += [None, None, None]
    fn = api.cover_attn_fwd if dt == "bf16" else api.cover_attn_fwd_f32
    out, lse = fn(*args)
    torch.cuda.synchronize()
    assert api.cover_device_status() == 0
    return out.float().cpu().numpy().astype(np.float64), lse.cpu().numpy().astype(np.float64)


def oracle_full(inp: W.AttnInputs):
    return oracle.override_attention(inp.as_f64("q"), inp.as_f64("k_cached"), inp.as_f64("v_cached"),
                                     inp.as_f64("k_seedmask"), inp.as_f64("v_seedmask"), inp.seed_idx)


def oracle_head_rows(inp: W.AttnInputs, b: int, hq: int, rows):
    """Oracle on one (b, hq) head, only the listed rows (one explicit view per row)."""
    G = inp.Hq // inp.Hkv
    hkv = hq // G
    cvt = W.bf16_bits_to_f64 if inp.dtype == "bf16" else (lambda a: a.astype(np.float64))
    q = cvt(inp.q[b:b + 1, hq:hq + 1])
    kc = cvt(inp.k_cached[b:b + 1, hkv:hkv + 1])
    vc = cvt(inp.v_cached[b:b + 1, hkv:hkv + 1])
    km = cvt(inp.k_seedmask[b:b + 1, hkv:hkv + 1])
    vm = cvt(inp.v_seedmask[b:b + 1, hkv:hkv + 1])
    return oracle.override_attention_rows(q, kc, vc, km, vm, inp.seed_idx[b:b + 1], 0, 0, rows)


def assert_bf16_close(out, ref, lse=None, ref_lse=None, what=""):
    d = np.abs(out - ref)
    assert d.max() <= TOL_BF16_MAX, f"{what} max |d| {d.max():.3e}"
    assert d.mean() <= TOL_BF16_MEAN, f"{what} mean |d| {d.mean():.3e}"
    if lse is not None:
        dl = np.abs(lse - ref_lse).max()
        assert dl <= TOL_LSE, f"{what} lse max |d| {dl:.3e}"


def assert_f32_close(out, ref, lse=None, ref_lse=None, what=""):
    d = np.abs(out - ref).max()
    assert d <= TOL_F32, f"{what} max |d| {d:.3e}"
    if lse is not None:
        dl = np.abs(lse - ref_lse).max()
        assert dl <= TOL_F32, f"{what} lse max |d| {dl:.3e}"
