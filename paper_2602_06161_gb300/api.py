"""Python binding of the COVER kernel library: same names as the C ABI.

Each function checks tensor dtypes / devices / contiguity, reads the sizes off
the tensors, and calls the C entry point on the current CUDA stream. All
arithmetic runs in the CUDA kernels; torch only provides device memory and
streams.
"""
from __future__ import annotations

import ctypes
from typing import Optional

import torch

from . import _lib


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else t.data_ptr()


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _need(t: torch.Tensor, name: str, dtype, ndim: int):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dims, got {tuple(t.shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def _attn(fn_name, dtype, q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx, out, lse, want_lse, stream):
    _need(q, "q", dtype, 4)
    _need(k_cached, "k_cached", dtype, 4)
    _need(v_cached, "v_cached", dtype, 4)
    B, Hq, L, D = q.shape
    Hkv = k_cached.shape[1]
    if tuple(k_cached.shape) != (B, Hkv, L, D) or tuple(v_cached.shape) != (B, Hkv, L, D):
        raise ValueError("k_cached / v_cached must be [B, Hkv, L, D] matching q")
    n_seeds = 0 if seed_idx is None else int(seed_idx.shape[1])
    if n_seeds > 0:
        _need(seed_idx, "seed_idx", torch.int32, 2)
        _need(k_seedmask, "k_seedmask", dtype, 4)
        _need(v_seedmask, "v_seedmask", dtype, 4)
        if tuple(seed_idx.shape) != (B, n_seeds):
            raise ValueError("seed_idx must be [B, S]")
        if tuple(k_seedmask.shape) != (B, Hkv, n_seeds, D) or tuple(v_seedmask.shape) != (B, Hkv, n_seeds, D):
            raise ValueError("k_seedmask / v_seedmask must be [B, Hkv, S, D]")
    if out is None:
        out = torch.empty_like(q)
    else:
        _need(out, "out", dtype, 4)
    if lse is None and want_lse:
        lse = torch.empty((B, Hq, L), dtype=torch.float32, device=q.device)
    elif lse is not None:
        _need(lse, "lse", torch.float32, 3)
    lib = _lib.load()
    code = getattr(lib, fn_name)(
        _ptr(q), _ptr(k_cached), _ptr(v_cached),
        _ptr(k_seedmask) if n_seeds else None, _ptr(v_seedmask) if n_seeds else None,
        _ptr(seed_idx) if n_seeds else None, n_seeds, B, Hq, Hkv, L, D,
        _ptr(out), _ptr(lse), _stream(stream))
    _lib.check(fn_name, code)
    return out, lse


def cover_attn_fwd(q, k_cached, v_cached, k_seedmask=None, v_seedmask=None, seed_idx=None, *,
                   out=None, lse=None, want_lse=True, stream=None):
    """Two-view override attention (bf16). Returns (out [B,Hq,L,D] bf16, lse [B,Hq,L] f32 or None)."""
    return _attn("cover_attn_fwd", torch.bfloat16, q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx,
                 out, lse, want_lse, stream)


def cover_attn_fwd_f32(q, k_cached, v_cached, k_seedmask=None, v_seedmask=None, seed_idx=None, *,
                       out=None, lse=None, want_lse=True, stream=None):
    """Two-view override attention in fp32 (CUDA cores)."""
    return _attn("cover_attn_fwd_f32", torch.float32, q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx,
                 out, lse, want_lse, stream)


def _attn_prefix(fn_name, dtype, q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx, q0, out, lse, want_lse,
                 stream, extra=()):
    _need(q, "q", dtype, 4)
    _need(k_cached, "k_cached", dtype, 4)
    _need(v_cached, "v_cached", dtype, 4)
    B, Hq, Lq, D = q.shape
    Hkv, Lk = k_cached.shape[1], k_cached.shape[2]
    if tuple(k_cached.shape) != (B, Hkv, Lk, D) or tuple(v_cached.shape) != (B, Hkv, Lk, D):
        raise ValueError("k_cached / v_cached must be [B, Hkv, Lk, D] matching q")
    n_seeds = 0 if seed_idx is None else int(seed_idx.shape[1])
    if n_seeds > 0:
        _need(seed_idx, "seed_idx", torch.int32, 2)
        _need(k_seedmask, "k_seedmask", dtype, 4)
        _need(v_seedmask, "v_seedmask", dtype, 4)
        if tuple(seed_idx.shape) != (B, n_seeds):
            raise ValueError("seed_idx must be [B, S]")
        if tuple(k_seedmask.shape) != (B, Hkv, n_seeds, D) or tuple(v_seedmask.shape) != (B, Hkv, n_seeds, D):
            raise ValueError("k_seedmask / v_seedmask must be [B, Hkv, S, D]")
    if out is None:
        out = torch.empty_like(q)
    else:
        _need(out, "out", dtype, 4)
    if lse is None and want_lse:
        lse = torch.empty((B, Hq, Lq), dtype=torch.float32, device=q.device)
    elif lse is not None:
        _need(lse, "lse", torch.float32, 3)
    code = getattr(_lib.load(), fn_name)(
        _ptr(q), _ptr(k_cached), _ptr(v_cached),
        _ptr(k_seedmask) if n_seeds else None, _ptr(v_seedmask) if n_seeds else None,
        _ptr(seed_idx) if n_seeds else None, n_seeds, B, Hq, Hkv, Lq, Lk, int(q0), D,
        _ptr(out), _ptr(lse), *extra, _stream(stream))
    _lib.check(fn_name, code)
    return out, lse


def cover_attn_fwd_prefix(q, k_cached, v_cached, k_seedmask=None, v_seedmask=None, seed_idx=None, *, q0: int,
                          out=None, lse=None, want_lse=True, stream=None):
    """Two-view attention for a window of Lq query rows at memory positions q0 .. q0+Lq-1 (bf16)."""
    return _attn_prefix("cover_attn_fwd_prefix", torch.bfloat16, q, k_cached, v_cached, k_seedmask, v_seedmask,
                        seed_idx, q0, out, lse, want_lse, stream)


def cover_attn_fwd_prefix_f32(q, k_cached, v_cached, k_seedmask=None, v_seedmask=None, seed_idx=None, *, q0: int,
                              out=None, lse=None, want_lse=True, stream=None):
    """The prefix-window attention in fp32 (CUDA cores)."""
    return _attn_prefix("cover_attn_fwd_prefix_f32", torch.float32, q, k_cached, v_cached, k_seedmask, v_seedmask,
                        seed_idx, q0, out, lse, want_lse, stream)


def _seed_route(fn_name, seed_idx, B, L, device, stream):
    n_seeds = 0 if seed_idx is None else int(seed_idx.shape[1])
    if n_seeds:
        _need(seed_idx, "seed_idx", torch.int32, 2)
        device = seed_idx.device
    device = device or torch.device("cuda")
    slot = torch.empty((B, L), dtype=torch.int32, device=device)
    bitmap = torch.empty((B, (L + 127) // 128, 4), dtype=torch.int32, device=device)
    n_invalid = torch.empty((1,), dtype=torch.int32, device=device)
    code = getattr(_lib.load(), fn_name)(_ptr(seed_idx) if n_seeds else None, n_seeds, B, L, _ptr(slot),
                                         _ptr(bitmap), _ptr(n_invalid), _stream(stream))
    _lib.check(fn_name, code)
    return slot, bitmap, n_invalid


def cover_seed_route(seed_idx: Optional[torch.Tensor], B: int, L: int, *, device=None, stream=None):
    """Seed routing as the kernels see it: (slot [B,L] int32, bitmap [B,ceil(L/128),4] int32 bits, n_invalid)."""
    return _seed_route("cover_seed_route", seed_idx, B, L, device, stream)


def cover_seed_route_debug(seed_idx: Optional[torch.Tensor], B: int, L: int, *, device=None, stream=None):
    """cover_seed_route under its boundary-table name (same C function behind it)."""
    return _seed_route("cover_seed_route_debug", seed_idx, B, L, device, stream)


def cover_score_workspace_bytes(n_seq: int) -> int:
    return int(_lib.load().cover_score_workspace_bytes(int(n_seq)))


def score_workspace(n_seq: int, device=None) -> torch.Tensor:
    """A zero-filled workspace for cover_score_fwd (reusable across calls on one stream)."""
    nbytes = cover_score_workspace_bytes(n_seq)
    return torch.zeros((max(nbytes, 4) + 3) // 4, dtype=torch.int32, device=device or "cuda")


def cover_score_fwd(logits, n_seq: int, topk: int, *, cur_tok=None, d_in=None, d_out=None, eligible=None,
                    workspace=None, out=None, stream=None):
    """Fused vocabulary scoring + per-segment top-k.

    Returns a dict of CUDA tensors: maxprob, entropy, argmax, score [N];
    topk_idx [n_seq, topk] int32 and topk_score [n_seq, topk] f32.
    """
    _need(logits, "logits", torch.bfloat16, 2)
    N, V = logits.shape
    dev = logits.device
    if cur_tok is not None:
        _need(cur_tok, "cur_tok", torch.int32, 1)
    if d_in is not None:
        _need(d_in, "d_in", torch.float32, 1)
    if d_out is not None:
        _need(d_out, "d_out", torch.float32, 1)
    if eligible is not None:
        _need(eligible, "eligible", torch.uint8, 1)
    if out is None:
        out = dict(
            maxprob=torch.empty(N, dtype=torch.float32, device=dev),
            entropy=torch.empty(N, dtype=torch.float32, device=dev),
            argmax=torch.empty(N, dtype=torch.int32, device=dev),
            score=torch.empty(N, dtype=torch.float32, device=dev),
            topk_idx=torch.empty((n_seq, max(topk, 0)), dtype=torch.int32, device=dev),
            topk_score=torch.empty((n_seq, max(topk, 0)), dtype=torch.float32, device=dev),
        )
    if workspace is None and topk > 0:
        workspace = score_workspace(n_seq, dev)
    code = _lib.load().cover_score_fwd(
        _ptr(logits), N, V, n_seq, _ptr(cur_tok), _ptr(d_in), _ptr(d_out), _ptr(eligible), topk,
        _ptr(out["maxprob"]), _ptr(out["entropy"]), _ptr(out["argmax"]), _ptr(out["score"]),
        _ptr(out["topk_idx"]) if topk > 0 else None, _ptr(out["topk_score"]) if topk > 0 else None,
        _ptr(workspace), _stream(stream))
    _lib.check("cover_score_fwd", code)
    return out


def cover_score_fwd_noalloc(logits, n_seq: int, topk: int, *, cur_tok=None, d_in=None, d_out=None, eligible=None,
                            out=None, stream=None):
    """cover_score_fwd without a workspace: for callers that cannot allocate device memory.

    The per-sequence counters live in a fixed device array of the library
    (at most 4096 sequences). Calls that overlap on the GPU race on that array.
    The first call on a device looks up the array's address; make it before
    any stream capture. Returns the same dict as cover_score_fwd.
    """
    _need(logits, "logits", torch.bfloat16, 2)
    N, V = logits.shape
    dev = logits.device
    for name, t, dt in (("cur_tok", cur_tok, torch.int32), ("d_in", d_in, torch.float32),
                        ("d_out", d_out, torch.float32), ("eligible", eligible, torch.uint8)):
        if t is not None:
            _need(t, name, dt, 1)
    if out is None:
        out = dict(
            maxprob=torch.empty(N, dtype=torch.float32, device=dev),
            entropy=torch.empty(N, dtype=torch.float32, device=dev),
            argmax=torch.empty(N, dtype=torch.int32, device=dev),
            score=torch.empty(N, dtype=torch.float32, device=dev),
            topk_idx=torch.empty((n_seq, max(topk, 0)), dtype=torch.int32, device=dev),
            topk_score=torch.empty((n_seq, max(topk, 0)), dtype=torch.float32, device=dev),
        )
    code = _lib.load().cover_score_fwd_noalloc(
        _ptr(logits), N, V, n_seq, _ptr(cur_tok), _ptr(d_in), _ptr(d_out), _ptr(eligible), topk,
        _ptr(out["maxprob"]), _ptr(out["entropy"]), _ptr(out["argmax"]), _ptr(out["score"]),
        _ptr(out["topk_idx"]) if topk > 0 else None, _ptr(out["topk_score"]) if topk > 0 else None,
        _stream(stream))
    _lib.check("cover_score_fwd_noalloc", code)
    return out


def _seed_kv(fn_name, k, v, seed_idx, k_cache, v_cache, stream):
    if k.dtype not in (torch.bfloat16, torch.float32):
        raise TypeError("k must be bfloat16 or float32")
    _need(k, "k", k.dtype, 4)
    _need(v, "v", k.dtype, 4)
    B, Hkv, L, D = k.shape
    if tuple(v.shape) != (B, Hkv, L, D):
        raise ValueError("v must match k")
    S = 0 if seed_idx is None else int(seed_idx.shape[1])
    if S > 0:
        _need(seed_idx, "seed_idx", torch.int32, 2)
        if tuple(seed_idx.shape) != (B, S):
            raise ValueError("seed_idx must be [B, S]")
        if k_cache is None:
            k_cache = torch.empty((B, Hkv, S, D), dtype=k.dtype, device=k.device)
            v_cache = torch.empty_like(k_cache)
        _need(k_cache, "k_cache", k.dtype, 4)
        _need(v_cache, "v_cache", k.dtype, 4)
        if tuple(k_cache.shape) != (B, Hkv, S, D) or tuple(v_cache.shape) != (B, Hkv, S, D):
            raise ValueError("k_cache / v_cache must be [B, Hkv, S, D]")
    code = getattr(_lib.load(), fn_name)(
        _ptr(k), _ptr(v), _ptr(seed_idx) if S else None, S, B, Hkv, L, D, k.element_size(),
        _ptr(k_cache) if S else None, _ptr(v_cache) if S else None, _stream(stream))
    _lib.check(fn_name, code)
    return k_cache, v_cache


def cover_seed_kv_gather(k, v, seed_idx, *, k_cache=None, v_cache=None, stream=None):
    """Cache the seeds' states at selection: returns (k_cache, v_cache) [B, Hkv, S, D]."""
    return _seed_kv("cover_seed_kv_gather", k, v, seed_idx, k_cache, v_cache, stream)


def cover_seed_kv_override(k, v, seed_idx, k_cache, v_cache, *, stream=None):
    """Swap the cached seed states into k, v (in place); the caches then hold the masked-input pairs."""
    if seed_idx is not None and seed_idx.shape[1] > 0 and (k_cache is None or v_cache is None):
        raise ValueError("k_cache and v_cache are required")
    return _seed_kv("cover_seed_kv_override", k, v, seed_idx, k_cache, v_cache, stream)


def cover_decide_workspace_bytes(N: int, n_seq: int) -> int:
    return int(_lib.load().cover_decide_workspace_bytes(int(N), int(n_seq)))


def decide_workspace(N: int, n_seq: int, device=None) -> torch.Tensor:
    """A zero-filled workspace for cover_score_decide_fwd (reusable across calls on one stream)."""
    nbytes = cover_decide_workspace_bytes(N, n_seq)
    return torch.zeros((max(nbytes, 16) + 15) // 16, 4, dtype=torch.int32, device=device or "cuda")


COVER_DECIDE_ALL = 0
COVER_DECIDE_UPDATE = 1


def cover_score_decide_fwd(logits, n_seq: int, tok, flags, remask_cnt, *, tau_draft: float, draft_budget: int,
                           remask_budget: int, mask_id: int, min_one: bool = True, pos0: int = 0,
                           max_seeds: int = 0, phase: int = COVER_DECIDE_ALL, d_in=None, d_out=None, draft_ok=None,
                           workspace=None, out=None, stream=None):
    """Scoring fused with one decoding step's decisions (drafting, revision, seed selection).

    tok (int32 [N]), flags and remask_cnt (uint8 [N]) are updated in place.
    Returns a dict of CUDA tensors: maxprob, entropy, argmax, score [N];
    seed_idx [n_seq, max_seeds] (positions, -1 padded), n_seeds [n_seq] and
    stats [n_seq, 6] (drafted, kept, replaced, remasked, n_t, n_above).
    With phase=COVER_DECIDE_UPDATE only drafting, revision and the state update
    run (score, seed_idx and n_seeds are left as they are); cover_attn_mass_fwd
    and cover_seed_select_fwd on the same workspace complete the step.
    """
    _need(logits, "logits", torch.bfloat16, 2)
    N, V = logits.shape
    dev = logits.device
    _need(tok, "tok", torch.int32, 1)
    _need(flags, "flags", torch.uint8, 1)
    _need(remask_cnt, "remask_cnt", torch.uint8, 1)
    for name, t, dt in (("d_in", d_in, torch.float32), ("d_out", d_out, torch.float32),
                        ("draft_ok", draft_ok, torch.uint8)):
        if t is not None:
            _need(t, name, dt, 1)
    if out is None:
        out = dict(
            maxprob=torch.empty(N, dtype=torch.float32, device=dev),
            entropy=torch.empty(N, dtype=torch.float32, device=dev),
            argmax=torch.empty(N, dtype=torch.int32, device=dev),
            score=torch.empty(N, dtype=torch.float32, device=dev),
            seed_idx=torch.empty((n_seq, max(max_seeds, 0)), dtype=torch.int32, device=dev),
            n_seeds=torch.empty(n_seq, dtype=torch.int32, device=dev),
            stats=torch.empty((n_seq, 6), dtype=torch.int32, device=dev),
        )
    if workspace is None:
        workspace = decide_workspace(N, n_seq, dev)
    code = _lib.load().cover_score_decide_fwd(
        _ptr(logits), N, V, n_seq, _ptr(d_in), _ptr(d_out), _ptr(draft_ok), float(tau_draft), int(draft_budget),
        int(remask_budget), int(mask_id), 1 if min_one else 0, int(pos0), int(max_seeds), int(phase),
        _ptr(tok), _ptr(flags), _ptr(remask_cnt), _ptr(out["maxprob"]), _ptr(out["entropy"]), _ptr(out["argmax"]),
        _ptr(out["score"]), _ptr(out["seed_idx"]) if max_seeds > 0 else None, _ptr(out["n_seeds"]),
        _ptr(out["stats"]), _ptr(workspace), _stream(stream))
    _lib.check("cover_score_decide_fwd", code)
    return out


def cover_seed_select_fwd(n_seq: int, tok, flags, remask_cnt, workspace, *, remask_budget: int, mask_id: int,
                          pos0: int = 0, max_seeds: int = 0, d_in=None, d_out=None, out=None, stream=None):
    """Seed score, adaptive revision rate and selection after a COVER_DECIDE_UPDATE call.

    `workspace` and the state tensors must be those of that call. Returns a
    dict of CUDA tensors: score [N], seed_idx [n_seq, max_seeds], n_seeds
    [n_seq], stats [n_seq, 6] (columns 4-5 written here).
    """
    _need(tok, "tok", torch.int32, 1)
    _need(flags, "flags", torch.uint8, 1)
    _need(remask_cnt, "remask_cnt", torch.uint8, 1)
    N = tok.shape[0]
    dev = tok.device
    for name, t in (("d_in", d_in), ("d_out", d_out)):
        if t is not None:
            _need(t, name, torch.float32, 1)
    if out is None:
        out = dict(score=torch.empty(N, dtype=torch.float32, device=dev),
                   seed_idx=torch.empty((n_seq, max(max_seeds, 0)), dtype=torch.int32, device=dev),
                   n_seeds=torch.empty(n_seq, dtype=torch.int32, device=dev),
                   stats=torch.zeros((n_seq, 6), dtype=torch.int32, device=dev))
    code = _lib.load().cover_seed_select_fwd(
        N, n_seq, _ptr(d_in), _ptr(d_out), int(remask_budget), int(mask_id), int(pos0), int(max_seeds),
        _ptr(tok), _ptr(flags), _ptr(remask_cnt), _ptr(out["score"]),
        _ptr(out["seed_idx"]) if max_seeds > 0 else None, _ptr(out["n_seeds"]), _ptr(out["stats"]),
        _ptr(workspace), _stream(stream))
    _lib.check("cover_seed_select_fwd", code)
    return out


def cover_attn_mass_workspace_bytes(B: int, Hq: int, per: int) -> int:
    return int(_lib.load().cover_attn_mass_workspace_bytes(int(B), int(Hq), int(per)))


def cover_attn_mass_fwd(q, k_cached, lse, tok, flags, *, mask_id: int, pos0: int, per: int, k_seedmask=None,
                        seed_idx=None, workspace=None, d_in=None, d_out=None, stream=None):
    """d_in / d_out (Section 5.3) of the response rows from the attention pass's q, K', lse.

    q [B, Hq, L, 128], k_cached [B, Hkv, L, 128] bf16, lse [B, Hq, L] f32 (as
    cover_attn_fwd wrote it), tok int32 / flags uint8 [B * per] (the state
    after a COVER_DECIDE_UPDATE call). Returns (d_in, d_out), float32 [B * per].
    """
    _need(q, "q", torch.bfloat16, 4)
    _need(k_cached, "k_cached", torch.bfloat16, 4)
    _need(lse, "lse", torch.float32, 3)
    _need(tok, "tok", torch.int32, 1)
    _need(flags, "flags", torch.uint8, 1)
    B, Hq, L, D = q.shape
    Hkv = k_cached.shape[1]
    n_seeds = 0 if seed_idx is None else int(seed_idx.shape[1])
    if n_seeds > 0:
        _need(seed_idx, "seed_idx", torch.int32, 2)
        _need(k_seedmask, "k_seedmask", torch.bfloat16, 4)
    if tok.shape[0] != B * per or flags.shape[0] != B * per:
        raise ValueError("tok / flags must have B * per entries")
    if workspace is None:
        nbytes = cover_attn_mass_workspace_bytes(B, Hq, per)
        workspace = torch.empty((nbytes + 15) // 16, 4, dtype=torch.int32, device=q.device)
    if d_in is None:
        d_in = torch.empty(B * per, dtype=torch.float32, device=q.device)
    if d_out is None:
        d_out = torch.empty(B * per, dtype=torch.float32, device=q.device)
    code = _lib.load().cover_attn_mass_fwd(
        _ptr(q), _ptr(k_cached), _ptr(k_seedmask) if n_seeds else None, _ptr(seed_idx) if n_seeds else None,
        n_seeds, _ptr(lse), B, Hq, Hkv, L, D, _ptr(tok), _ptr(flags), int(mask_id), int(pos0), int(per),
        _ptr(workspace), _ptr(d_in), _ptr(d_out), _stream(stream))
    _lib.check("cover_attn_mass_fwd", code)
    return d_in, d_out


def cover_device_status(stream=None) -> int:
    """Synchronise the stream; return and clear the device status word (0 = OK)."""
    return int(_lib.load().cover_device_status(_stream(stream)))


def cover_status_str(code: int) -> str:
    return _lib.status_str(code)


def cover_debug_umma_tile(a, b, p, v, *, stream=None):
    for name, t in (("a", a), ("b", b), ("p", p), ("v", v)):
        _need(t, name, torch.bfloat16, 2)
        if tuple(t.shape) != (128, 128):
            raise ValueError(f"{name} must be [128, 128]")
    c1 = torch.empty((128, 128), dtype=torch.float32, device=a.device)
    c2 = torch.empty((128, 128), dtype=torch.float32, device=a.device)
    code = _lib.load().cover_debug_umma_tile(_ptr(a), _ptr(b), _ptr(p), _ptr(v), _ptr(c1), _ptr(c2),
                                             _stream(stream))
    _lib.check("cover_debug_umma_tile", code)
    return c1, c2


def cover_debug_wait_timeout(limit_us: int, *, stream=None) -> None:
    _lib.check("cover_debug_wait_timeout", _lib.load().cover_debug_wait_timeout(int(limit_us), _stream(stream)))


def cover_debug_attn_prefix_packed(q, k_cached, v_cached, k_seedmask=None, v_seedmask=None, seed_idx=None, *,
                                   q0: int, fault_cta: int = -1, limit_us: int = 0, out=None, lse=None,
                                   want_lse=True, stream=None):
    """The prefix-window attention (bf16) on the packed grouped-query window kernel, whichever kernel
    cover_attn_fwd_prefix would pick for the shape; fault_cta >= 0 or limit_us > 0 run its self-test
    instance (CTA fault_cta leaves out its first K load, waits give up after limit_us)."""
    return _attn_prefix("cover_debug_attn_prefix_packed", torch.bfloat16, q, k_cached, v_cached, k_seedmask,
                        v_seedmask, seed_idx, q0, out, lse, want_lse, stream,
                        extra=(int(fault_cta), int(limit_us)))


def cover_debug_attn_fault(q, k_cached, v_cached, k_seedmask=None, v_seedmask=None, seed_idx=None, *, q0: int = 0,
                           fault_cta: int, fault_entry: int, limit_us: int, out=None, lse=None, stream=None):
    """Self-test: the bf16 attention (window form) with CTA fault_cta leaving out one K tile load and every
    bounded wait limited to limit_us; read the outcome with cover_debug_status_detail()."""
    return _attn_prefix("cover_debug_attn_fault", torch.bfloat16, q, k_cached, v_cached, k_seedmask, v_seedmask,
                        seed_idx, q0, out, lse, True, stream,
                        extra=(int(fault_cta), int(fault_entry), int(limit_us)))


def cover_debug_window_model(B: int, Hq: int, Hkv: int, Lq: int, Lk: int, q0: int, n_sm: int, max_clusters):
    """The prefix-window call's choice between the packed grouped-query kernel and the square kernel
    on a GPU with n_sm SMs and max_clusters[c - 1] resident clusters of c packed CTAs (c = 1 .. 8).
    Host arithmetic only (no device needed)."""
    mc = (ctypes.c_int32 * 8)(*[int(x) for x in max_clusters])
    choice = (ctypes.c_int32 * 6)()
    times = (ctypes.c_double * 2)()
    _lib.check("cover_debug_window_model",
               _lib.load().cover_debug_window_model(B, Hq, Hkv, Lq, Lk, q0, n_sm, mc, choice, times))
    return {"supported": bool(choice[0]), "resident": bool(choice[1]), "packed": bool(choice[2]),
            "T": int(choice[3]), "nsplit": int(choice[4]), "n_qt": int(choice[5]),
            "packed_us": float(times[0]), "square_us": float(times[1])}


def cover_debug_status_detail(stream=None):
    """(status code, site id, block id) of the current device's status block, which is then cleared."""
    detail = (ctypes.c_int32 * 3)()
    _lib.check("cover_debug_status_detail", _lib.load().cover_debug_status_detail(detail, _stream(stream)))
    return int(detail[0]), int(detail[1]), int(detail[2])
