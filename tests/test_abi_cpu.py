"""CPU checks of the C-ABI library: it builds, loads without a GPU, exports every
declared symbol, and rejects invalid arguments before touching CUDA."""
import ctypes
import os
import re

import pytest

from paper_2602_06161_gb300 import _lib, build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = []
    for h in sorted(os.listdir(os.path.join(ROOT, "include"))):
        if h.endswith(".h"):
            text = open(os.path.join(ROOT, "include", h)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names += re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\**\s*(cover_[A-Za-z0-9_]+)\s*\(",
                                text, flags=re.M)
    return names


@pytest.fixture(scope="module")
def lib():
    build.build()
    return _lib.load()


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 9
    raw = ctypes.CDLL(build.LIB)
    for n in names:
        assert hasattr(raw, n), n
    assert sorted(names) == sorted(_lib.exported_symbols())


def test_status_strings(lib):
    assert _lib.status_str(0) == "COVER_OK"
    assert _lib.status_str(-1) == "COVER_ERR_INVALID_ARG"
    assert _lib.status_str(-4) == "COVER_ERR_DEVICE_TIMEOUT"
    assert _lib.status_str(12345) == "COVER_ERR_UNKNOWN"


# fake, 16-byte aligned, never dereferenced (argument checks return first)
P = 0x10000


def attn(lib, **kw):
    a = dict(q=P, kc=P, vc=P, km=P, vm=P, seeds=P, S=2, B=1, Hq=2, Hkv=1, L=128, D=128, out=P, lse=P)
    a.update(kw)
    return lib.cover_attn_fwd(a["q"], a["kc"], a["vc"], a["km"], a["vm"], a["seeds"], a["S"], a["B"], a["Hq"],
                              a["Hkv"], a["L"], a["D"], a["out"], a["lse"], None)


@pytest.mark.parametrize("kw", [
    dict(q=None), dict(out=None), dict(kc=None), dict(B=0), dict(L=0), dict(Hq=3, Hkv=2), dict(Hkv=0),
    dict(S=-1), dict(S=129), dict(seeds=None), dict(km=None), dict(q=P + 8), dict(out=P + 2), dict(lse=P + 2),
    dict(D=0),
])
def test_attn_invalid_args(lib, kw):
    assert attn(lib, **kw) == -1


def test_attn_unsupported_head_dim(lib):
    assert attn(lib, D=64) == -2
    assert attn(lib, D=96) == -2


def score(lib, **kw):
    a = dict(logits=P, N=8, V=16, n_seq=2, k=2, mp=P, ent=P, am=P, sc=P, ti=P, ts=P, ws=P)
    a.update(kw)
    return lib.cover_score_fwd(a["logits"], a["N"], a["V"], a["n_seq"], None, None, None, None, a["k"], a["mp"],
                               a["ent"], a["am"], a["sc"], a["ti"], a["ts"], a["ws"], None)


@pytest.mark.parametrize("kw", [
    dict(logits=None), dict(N=0), dict(V=0), dict(n_seq=3), dict(n_seq=0), dict(k=5), dict(k=-1),
    dict(ti=None), dict(ws=None), dict(logits=P + 2), dict(mp=None), dict(N=2 * 4097, n_seq=2),
])
def test_score_invalid_args(lib, kw):
    assert score(lib, **kw) == -1


@pytest.mark.parametrize("name", ["cover_seed_route", "cover_seed_route_debug"])
def test_route_invalid_args(lib, name):
    fn = getattr(lib, name)
    assert fn(P, 2, 0, 10, P, P, P, None) == -1
    assert fn(P, 11, 1, 10, P, P, P, None) == -1
    assert fn(None, 2, 1, 10, P, P, P, None) == -1
    assert fn(P, 2, 1, 10, None, P, P, None) == -1


def test_boundary_names_exported(lib):
    # the entry points the boundary's specification names, under those names
    raw = ctypes.CDLL(build.LIB)
    for n in ["cover_attn_fwd", "cover_attn_fwd_f32", "cover_score_fwd", "cover_seed_route_debug",
              "cover_device_status", "cover_status_str"]:
        assert hasattr(raw, n), n


def test_debug_invalid_args(lib):
    assert lib.cover_debug_wait_timeout(0, None) == -1
    assert lib.cover_debug_wait_timeout(3000000, None) == -1
    assert lib.cover_debug_umma_tile(None, P, P, P, P, P, None) == -1


def test_workspace_bytes(lib):
    assert lib.cover_score_workspace_bytes(8) == 32
    assert lib.cover_score_workspace_bytes(0) == 0


def decide(lib, **kw):
    a = dict(logits=P, N=8, V=32, n_seq=2, d_in=None, d_out=None, draft_ok=None, tau=0.8, budget=2, remask_budget=3,
             mask_id=31, min_one=1, pos0=0, max_seeds=4, phase=0, tok=P, flags=P, remask_cnt=P, maxprob=P, entropy=P,
             argmax=P, score=P, seed_idx=P, n_seeds=P, stats=None, workspace=P)
    a.update(kw)
    return lib.cover_score_decide_fwd(*a.values(), None)


@pytest.mark.parametrize("kw", [
    dict(logits=None), dict(tok=None), dict(flags=None), dict(remask_cnt=None), dict(n_seeds=None),
    dict(workspace=None), dict(N=0), dict(V=0), dict(n_seq=3), dict(N=8194, n_seq=2), dict(budget=-1),
    dict(remask_budget=-1), dict(max_seeds=-1), dict(seed_idx=None), dict(logits=P + 2), dict(workspace=P + 4),
    dict(tok=P + 2), dict(phase=2), dict(phase=-1),
])
def test_decide_invalid_args(lib, kw):
    assert decide(lib, **kw) == -1


def test_decide_workspace_bytes(lib):
    assert lib.cover_decide_workspace_bytes(8, 2) == 16 + 64
    assert lib.cover_decide_workspace_bytes(4096, 5) == 32 + 8 * 4096
    assert lib.cover_decide_workspace_bytes(0, 1) == 0


@pytest.mark.parametrize("fn", ["cover_seed_kv_gather", "cover_seed_kv_override"])
@pytest.mark.parametrize("kw", [
    dict(k=None), dict(v=None), dict(B=0), dict(Hkv=0), dict(L=0), dict(D=0), dict(n_seeds=-1),
    dict(elem_bytes=1), dict(elem_bytes=8), dict(D=4), dict(D=65536), dict(seed_idx=None), dict(k_cache=None),
    dict(v_cache=None), dict(k=P + 8), dict(k_cache=P + 8), dict(seed_idx=P + 2),
])
def test_seed_kv_invalid_args(lib, fn, kw):
    a = dict(k=P, v=P, seed_idx=P, n_seeds=4, B=2, Hkv=2, L=16, D=128, elem_bytes=2, k_cache=P, v_cache=P)
    a.update(kw)
    assert getattr(lib, fn)(*a.values(), None) == -1


def test_seed_kv_no_seeds_is_a_noop(lib):
    # nothing to move: returns before touching the device
    assert lib.cover_seed_kv_override(P, P, None, 0, 2, 2, 16, 128, 2, None, None, None) == 0
    assert lib.cover_seed_kv_gather(P, P, None, 0, 2, 2, 16, 128, 2, None, None, None) == 0


@pytest.mark.parametrize("fn", ["cover_attn_fwd_prefix", "cover_attn_fwd_prefix_f32"])
@pytest.mark.parametrize("kw", [
    dict(Lq=0), dict(Lk=0), dict(q0=-1), dict(q0=50, Lq=51), dict(n_seeds=101), dict(q=None), dict(Hq=3),
])
def test_prefix_invalid_args(lib, fn, kw):
    a = dict(q=P, kc=P, vc=P, km=P, vm=P, seeds=P, n_seeds=4, B=1, Hq=4, Hkv=2, Lq=50, Lk=100, q0=50, D=128,
             out=P, lse=None)
    a.update(kw)
    assert getattr(lib, fn)(*a.values(), None) == -1


def test_prefix_unsupported_head_dim(lib):
    assert lib.cover_attn_fwd_prefix(P, P, P, P, P, P, 4, 1, 4, 2, 50, 100, 50, 64, P, None, None) == -2


@pytest.mark.parametrize("kw", [
    dict(tok=None), dict(flags=None), dict(rc=None), dict(score=None), dict(n_seeds=None), dict(ws=None),
    dict(N=0), dict(n_seq=3), dict(N=8194, n_seq=2), dict(remask_budget=-1), dict(max_seeds=-1),
    dict(seed_idx=None), dict(ws=P + 4),
])
def test_select_invalid_args(lib, kw):
    a = dict(N=8, n_seq=2, d_in=None, d_out=None, remask_budget=3, mask_id=31, pos0=0, max_seeds=4, tok=P, flags=P,
             rc=P, score=P, seed_idx=P, n_seeds=P, stats=None, ws=P)
    a.update(kw)
    assert lib.cover_seed_select_fwd(*a.values(), None) == -1


@pytest.mark.parametrize("kw", [
    dict(q=None), dict(lse=None), dict(tok=None), dict(ws=None), dict(d_in=None), dict(B=0), dict(Hq=3),
    dict(per=0), dict(pos0=-1), dict(pos0=10, per=7), dict(n_seeds=17), dict(seed_idx=None), dict(q=P + 8),
])
def test_mass_invalid_args(lib, kw):
    a = dict(q=P, k=P, km=P, seed_idx=P, n_seeds=2, lse=P, B=1, Hq=4, Hkv=2, L=16, D=128, tok=P, flags=P,
             mask_id=9, pos0=8, per=8, ws=P, d_in=P, d_out=P)
    a.update(kw)
    assert lib.cover_attn_mass_fwd(*a.values(), None) == -1


def test_mass_unsupported_head_dim(lib):
    assert lib.cover_attn_mass_fwd(P, P, P, P, 2, P, 1, 4, 2, 16, 64, P, P, 9, 8, 8, P, P, P, None) == -2


def test_mass_unsupported_block_length(lib):
    # a response block longer than the shared-memory staging holds
    L = 20000
    assert lib.cover_attn_mass_fwd(P, P, P, P, 2, P, 1, 4, 2, L, 128, P, P, 9, 0, 16385, P, P, P, None) == -2
