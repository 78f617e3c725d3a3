"""Seeded synthetic PCED workloads: shapes, cache lengths, retrieval scores and
the bf16 tensors (KV-cache prefixes, token embedding, unembedding weights).

This module defines inputs only and holds none of the decoding method's
arithmetic.  The CPU oracle (``oracle/``) and the CUDA path
(``paper_2601_08670_gb300``) both take their inputs from here.

Recipe (the paper runs real LLMs on LOFT / LongBench documents, Sec. 4 and
App. A; no weights or datasets are used here, so these seeded tensors stand in
for them with the paper's model shapes):
  * K/V cache prefix elements ~ N(0, 1), bf16; one counter-based stream per
    (tensor, layer, sequence, kv-head), element index = position * D + dim.
  * token embedding E[V, d] ~ N(0, 1), unembedding W_U[V, d] ~ N(0, 0.02^2).
  * cache lengths: per workload (fixed, uniform, or clipped normal document
    lengths plus 32 query tokens; the amateur holds the 32 query tokens only,
    following App. A: the amateur is the system prompt plus the shared question
    template).
  * retrieval scores r in (0, 1]: U[0,1], softmax of N(0, 2^2) logits, flat 0.5,
    or one-hot-ish 0.95 / 0.01.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
from dataclasses import dataclass, field, replace

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIBDIR = os.path.join(HERE, "_lib")

T_KCACHE, T_VCACHE, T_EMBED, T_UNEMBED = 1, 2, 3, 4
SIGMA_KV, SIGMA_EMBED, SIGMA_UNEMBED = 1.0, 1.0, 0.02


def normal_scale(sigma: float) -> float:
    """fp32 multiplier turning the centred Irwin-Hall(4) integer into N(0, sigma^2)."""
    return float(np.float32(sigma * math.sqrt(3.0) / 65536.0))


# --------------------------------------------------------------------------
# workloads
# --------------------------------------------------------------------------
@dataclass(frozen=True)
class Workload:
    name: str
    B: int          # independent queries
    N: int          # document experts per query (the amateur is extra)
    L: int          # layers
    Hq: int
    Hkv: int
    D: int
    V: int
    steps: int
    doc_len: tuple  # ("fixed", n) | ("uniform", lo, hi) | ("clipnormal", mu, sd, lo, hi)
    query_tokens: int = 32
    amateur_len: int = 32
    r_recipe: tuple = ("uniform",)
    beta: float = 0.5
    gamma: float = 2.5
    seed: int = 0
    bos: int = 0
    description: str = ""

    @property
    def d(self) -> int:
        return self.Hq * self.D

    @property
    def S(self) -> int:
        return self.B * (self.N + 1)

    @property
    def G(self) -> int:
        return self.Hq // self.Hkv


WORKLOADS = {
    "tiny": Workload(
        "tiny", B=1, N=2, L=1, Hq=8, Hkv=2, D=64, V=8192, steps=4,
        doc_len=("fixed", 256), query_tokens=0, amateur_len=32,
        description="tiny PCED step: N=2 doc experts + amateur, 1 layer (8 q / 2 kv heads, head_dim 64, "
                    "hidden 512), vocab 8192, doc KV 256, amateur KV 32, 4 greedy steps"),
    "llama8": Workload(
        "llama8", B=1, N=8, L=32, Hq=32, Hkv=8, D=128, V=128256, steps=64,
        doc_len=("fixed", 2048),
        description="Llama-3-8B shapes, N=8 doc experts + amateur, doc KV 2048+32, vocab 128256, 64 steps"),
    "llama8_l4": Workload(
        "llama8_l4", B=1, N=8, L=4, Hq=32, Hkv=8, D=128, V=128256, steps=16,
        doc_len=("fixed", 2048),
        description="llama8 with 4 layers: the same per-layer work, small enough for multi-pass profiling"),
    "llama32": Workload(
        "llama32", B=1, N=32, L=32, Hq=32, Hkv=8, D=128, V=128256, steps=64,
        doc_len=("uniform", 512, 8192), r_recipe=("softmax_normal", 2.0),
        description="Llama-3-8B shapes, N=32 doc experts + amateur, ragged doc KV U[512,8192]+32, "
                    "r = softmax(N(0,2^2)), 64 steps"),
    "manydoc": Workload(
        "manydoc", B=16, N=16, L=32, Hq=32, Hkv=8, D=128, V=128256, steps=32,
        doc_len=("clipnormal", 1024.0, 256.0, 256, 2048),
        description="16 queries x (16 doc experts + amateur) = 272 sequences, doc KV N(1024,256) clipped "
                    "[256,2048]+32, Llama-3-8B shapes, 32 steps"),
    "llama8_k64": Workload(
        "llama8_k64", B=1, N=64, L=32, Hq=32, Hkv=8, D=128, V=128256, steps=16,
        doc_len=("fixed", 2048),
        description="Llama-3-8B shapes, top-k = 64 doc experts of KV 2048+32 + amateur, vocab 128256, 16 steps"),
    "llama8_k128": Workload(
        "llama8_k128", B=1, N=128, L=32, Hq=32, Hkv=8, D=128, V=128256, steps=16,
        doc_len=("fixed", 2048),
        description="Llama-3-8B shapes, top-k = 128 doc experts of KV 2048+32 + amateur, vocab 128256, 16 steps"),
    "qwen_flat": Workload(
        "qwen_flat", B=1, N=16, L=28, Hq=28, Hkv=4, D=128, V=151936, steps=128,
        doc_len=("fixed", 4096), r_recipe=("flat", 0.5),
        description="Qwen2-7B shapes, N=16 doc experts of KV 4096+32, flat retrieval scores 0.5, 128 steps"),
    "qwen_onehot": Workload(
        "qwen_onehot", B=1, N=16, L=28, Hq=28, Hkv=4, D=128, V=151936, steps=128,
        doc_len=("fixed", 4096), r_recipe=("onehot", 0.95, 0.01),
        description="Qwen2-7B shapes, N=16 doc experts of KV 4096+32, one-hot-ish scores 0.95/0.01, 128 steps"),
}


def get(name: str, **overrides) -> Workload:
    w = WORKLOADS[name]
    return replace(w, **overrides) if overrides else w


def base_lengths(w: Workload) -> np.ndarray:
    """Cache length of every sequence before the first decode step, [S] int32.
    Sequence order is query-major; the amateur is first within a query."""
    rng = np.random.default_rng([w.seed, 1])
    kind = w.doc_len[0]
    n_docs = w.B * w.N
    if kind == "fixed":
        docs = np.full(n_docs, w.doc_len[1], dtype=np.int64)
    elif kind == "uniform":
        docs = rng.integers(w.doc_len[1], w.doc_len[2], endpoint=True, size=n_docs)
    elif kind == "clipnormal":
        mu, sd, lo, hi = w.doc_len[1:]
        docs = np.clip(np.rint(rng.normal(mu, sd, size=n_docs)), lo, hi).astype(np.int64)
    else:
        raise ValueError(kind)
    docs = docs + w.query_tokens
    out = np.empty(w.S, dtype=np.int32)
    for b in range(w.B):
        out[b * (w.N + 1)] = w.amateur_len
        out[b * (w.N + 1) + 1:(b + 1) * (w.N + 1)] = docs[b * w.N:(b + 1) * w.N]
    return out


def retrieval_scores(w: Workload) -> np.ndarray:
    """Fused relevance scores r_k in (0, 1], [B, N] fp32."""
    rng = np.random.default_rng([w.seed, 2])
    kind = w.r_recipe[0]
    if kind == "uniform":
        r = rng.uniform(0.0, 1.0, size=(w.B, w.N))
    elif kind == "softmax_normal":
        z = rng.normal(0.0, w.r_recipe[1], size=(w.B, w.N))
        z = z - z.max(axis=1, keepdims=True)
        r = np.exp(z) / np.exp(z).sum(axis=1, keepdims=True)
    elif kind == "flat":
        r = np.full((w.B, w.N), w.r_recipe[1])
    elif kind == "onehot":
        hi, lo = w.r_recipe[1], w.r_recipe[2]
        r = np.full((w.B, w.N), lo)
        idx = rng.integers(0, w.N, size=w.B)
        r[np.arange(w.B), idx] = hi
    else:
        raise ValueError(kind)
    return r.astype(np.float32)


def betas(w: Workload) -> np.ndarray:
    """Per-expert contrastive strength (a fixed beta_0 broadcast), [B, N] fp32."""
    return np.full((w.B, w.N), w.beta, dtype=np.float32)


@dataclass
class CacheLayout:
    """Geometry of the KV caches.  Slab (layer l, sequence s, kv-head h) starts
    at element l*layer_elems + kv_offset[s] + h*cap[s]*D and holds cap[s]
    rows of D bf16 elements."""
    cap: np.ndarray        # [S] int32
    kv_offset: np.ndarray  # [S] int64
    layer_elems: int
    L: int
    Hkv: int
    D: int

    @property
    def total_elems(self) -> int:
        return self.L * self.layer_elems


def cache_layout(w: Workload, base_len: np.ndarray, extra: int | None = None) -> CacheLayout:
    extra = w.steps if extra is None else extra
    cap = (base_len.astype(np.int64) + extra).astype(np.int32)
    sizes = w.Hkv * cap.astype(np.int64) * w.D
    off = np.zeros(len(cap), dtype=np.int64)
    off[1:] = np.cumsum(sizes)[:-1]
    return CacheLayout(cap=cap, kv_offset=off, layer_elems=int(sizes.sum()), L=w.L, Hkv=w.Hkv, D=w.D)


@dataclass
class PagedLayout:
    """Paged KV layout: each layer's pool is num_blocks blocks of [Hkv][P][D];
    row pos of (sequence s, kv-head h) lives in block table[s][pos // P], row
    pos % P.  Blocks are handed out in a seeded random order (a serving
    allocator's scattered pages)."""
    P: int
    table: np.ndarray      # [S][max_blocks] int32 (-1 past a sequence's blocks)
    num_blocks: int
    cap: np.ndarray        # [S] int32 logical capacity (rows)
    layer_elems: int
    L: int
    Hkv: int
    D: int

    @property
    def max_blocks(self) -> int:
        return int(self.table.shape[1])

    @property
    def total_elems(self) -> int:
        return self.L * self.layer_elems


def paged_layout(w: Workload, base_len: np.ndarray, P: int, extra: int | None = None) -> PagedLayout:
    extra = w.steps if extra is None else extra
    cap = (base_len.astype(np.int64) + extra).astype(np.int32)
    nblk = (cap.astype(np.int64) + P - 1) // P
    num_blocks = int(nblk.sum())
    order = np.random.default_rng([w.seed, 0x9A6E]).permutation(num_blocks).astype(np.int32)
    table = np.full((len(cap), int(nblk.max())), -1, np.int32)
    at = 0
    for s, n in enumerate(nblk):
        table[s, :n] = order[at:at + n]
        at += n
    return PagedLayout(P=P, table=table, num_blocks=num_blocks, cap=cap,
                       layer_elems=num_blocks * w.Hkv * P * w.D, L=w.L, Hkv=w.Hkv, D=w.D)


def kv_bytes_per_token(L: int, Hkv: int, D: int, elem_bytes: int = 2) -> int:
    """K and V bytes one token occupies across all layers."""
    return L * 2 * Hkv * D * elem_bytes


def algorithmic_bytes_per_step(w: Workload, lens: np.ndarray) -> int:
    """Bytes one decode step must read: every cached K/V row of every layer
    (lens counts the token appended this step) plus the unembedding matrix."""
    return int(np.sum(lens.astype(np.int64))) * kv_bytes_per_token(w.L, w.Hkv, w.D) + w.V * w.d * 2


# --------------------------------------------------------------------------
# native fills
# --------------------------------------------------------------------------
def _build_host(force: bool = False) -> str:
    os.makedirs(LIBDIR, exist_ok=True)
    so = os.path.join(LIBDIR, "libsynth_host.so")
    src = os.path.join(HERE, "synth_host.c")
    if force or not os.path.exists(so) or os.path.getmtime(so) < max(
            os.path.getmtime(src), os.path.getmtime(os.path.join(HERE, "synth.h"))):
        tmp = so + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fPIC", "-shared", "-ffp-contract=off", "-pthread",
                               "-o", tmp, src])
        os.replace(tmp, so)
    return so


def _build_dev(force: bool = False) -> str:
    os.makedirs(LIBDIR, exist_ok=True)
    so = os.path.join(LIBDIR, "libsynth_dev.so")
    src = os.path.join(HERE, "synth_dev.cu")
    if force or not os.path.exists(so) or os.path.getmtime(so) < max(
            os.path.getmtime(src), os.path.getmtime(os.path.join(HERE, "synth.h"))):
        tmp = so + f".tmp{os.getpid()}"
        subprocess.check_call(["nvcc", "-O3", "-shared", "-Xcompiler", "-fPIC", "-fmad=false",
                               "-gencode", "arch=compute_103a,code=sm_103a", "-o", tmp, src])
        os.replace(tmp, so)
    return so


def build(force: bool = False) -> None:
    _build_host(force)
    _build_dev(force)


_host = None
_dev = None


def host_lib():
    global _host
    if _host is None:
        lib = ctypes.CDLL(_build_host())
        P, I64, I32, U64, U32, F = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_uint64,
                                    ctypes.c_uint32, ctypes.c_float)
        lib.synth_fill_cache.argtypes = [P, I64, P, P, P, P, I32, I32, I32, I32, U64, U32, F, I32]
        lib.synth_fill_cache.restype = None
        lib.synth_fill_matrix.argtypes = [P, I64, I64, I64, U64, U32, F, I32]
        lib.synth_fill_matrix.restype = None
        lib.synth_key.argtypes = [U64, U32, U32, U32, U32]
        lib.synth_key.restype = U64
        lib.synth_value_bf16.argtypes = [U64, U64, F]
        lib.synth_value_bf16.restype = ctypes.c_uint16
        lib.synth_value_f32.argtypes = [U64, U64, F]
        lib.synth_value_f32.restype = F
        _host = lib
    return _host


def dev_lib():
    global _dev
    if _dev is None:
        lib = ctypes.CDLL(_build_dev())
        P, I64, I32, U64, U32, F = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_uint64,
                                    ctypes.c_uint32, ctypes.c_float)
        lib.synth_dev_fill_cache.argtypes = [P, I64, P, P, P, P, I32, I32, I32, I32, U64, U32, F, P]
        lib.synth_dev_fill_cache.restype = ctypes.c_int
        lib.synth_dev_fill_cache_paged.argtypes = [P, I64, P, I32, I32, P, P, I32, I32, I32, I32, U64, U32, F, P]
        lib.synth_dev_fill_cache_paged.restype = ctypes.c_int
        lib.synth_dev_fill_matrix.argtypes = [P, I64, I64, I64, U64, U32, F, P]
        lib.synth_dev_fill_matrix.restype = ctypes.c_int
        _dev = lib
    return _dev


def _threads() -> int:
    return max(1, min(64, os.cpu_count() or 1))


def _ptr(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


def host_matrix(w: Workload, tensor: int, row0: int = 0, rows: int | None = None) -> np.ndarray:
    """Rows [row0, row0+rows) of the embedding (T_EMBED) or unembedding
    (T_UNEMBED) matrix as bf16 bit patterns, uint16 [rows, d]."""
    rows = w.V - row0 if rows is None else rows
    sigma = SIGMA_EMBED if tensor == T_EMBED else SIGMA_UNEMBED
    out = np.empty((rows, w.d), dtype=np.uint16)
    host_lib().synth_fill_matrix(_ptr(out), row0, rows, w.d, w.seed, tensor, normal_scale(sigma), _threads())
    return out


def host_caches(w: Workload, layout: CacheLayout, base_len: np.ndarray, seq_ids: np.ndarray | None = None):
    """K and V caches (bf16 bit patterns, uint16 [L * layer_elems]) with the
    generated prefixes filled in and zeros after them."""
    S = len(base_len)
    seq_ids = np.arange(S, dtype=np.int32) if seq_ids is None else np.ascontiguousarray(seq_ids, dtype=np.int32)
    base_len = np.ascontiguousarray(base_len, dtype=np.int32)
    cap = np.ascontiguousarray(layout.cap, dtype=np.int32)
    off = np.ascontiguousarray(layout.kv_offset, dtype=np.int64)
    out = []
    for tensor in (T_KCACHE, T_VCACHE):
        c = np.zeros(layout.total_elems, dtype=np.uint16)
        host_lib().synth_fill_cache(_ptr(c), layout.layer_elems, _ptr(off), _ptr(cap), _ptr(base_len),
                                    _ptr(seq_ids), S, w.L, w.Hkv, w.D, w.seed, tensor,
                                    normal_scale(SIGMA_KV), _threads())
        out.append(c)
    return out[0], out[1]


def dev_fill_caches(w: Workload, layer_elems: int, k_cache, v_cache, kv_offset_dev, cap_dev, base_len_dev,
                    seq_ids_dev, stream_ptr: int):
    """Fill device caches (torch tensors) exactly like host_caches."""
    S = int(base_len_dev.numel())
    for tensor, buf in ((T_KCACHE, k_cache), (T_VCACHE, v_cache)):
        rc = dev_lib().synth_dev_fill_cache(buf.data_ptr(), int(layer_elems), kv_offset_dev.data_ptr(),
                                            cap_dev.data_ptr(), base_len_dev.data_ptr(), seq_ids_dev.data_ptr(),
                                            S, w.L, w.Hkv, w.D, w.seed, tensor, normal_scale(SIGMA_KV), stream_ptr)
        if rc != 0:
            raise RuntimeError(f"synth_dev_fill_cache failed: cuda error {rc}")


def dev_fill_matrix(w: Workload, tensor: int, out, stream_ptr, row0: int = 0, rows: int | None = None):
    rows = w.V - row0 if rows is None else rows
    sigma = SIGMA_EMBED if tensor == T_EMBED else SIGMA_UNEMBED
    rc = dev_lib().synth_dev_fill_matrix(out.data_ptr(), row0, rows, w.d, w.seed, tensor,
                                         normal_scale(sigma), stream_ptr)
    if rc != 0:
        raise RuntimeError(f"synth_dev_fill_matrix failed: cuda error {rc}")


T_MISC = 9


def host_normal_bf16(n: int, seed: int, sigma: float = 1.0) -> np.ndarray:
    """n bf16 samples (bit patterns) of an auxiliary stream, for test operands."""
    out = np.empty(n, dtype=np.uint16)
    host_lib().synth_fill_matrix(_ptr(out), 0, 1, n, seed, T_MISC, normal_scale(sigma), _threads())
    return out


def expert_part(w: Workload, e0: int, e1: int):
    """The sequences of every query's amateur and contextual experts
    [e0, e1) (0-based): the workload with N = e1 - e0, the global sequence
    ids (query-major, amateur first) and the columns of beta / r."""
    assert 0 <= e0 < e1 <= w.N
    ids = np.array([b * (w.N + 1) + j for b in range(w.B) for j in [0] + list(range(1 + e0, 1 + e1))], np.int32)
    return replace(w, N=e1 - e0), ids, slice(e0, e1)


def device_inputs(w: Workload, device="cuda", extra_steps: int | None = None, stream=None,
                  paged: int = 0, part: tuple | None = None) -> dict:
    """All inputs of workload `w` as device tensors: caches with generated
    prefixes (zeros after), embedding, unembedding, lengths, layout tables,
    beta and r.  Generated on the device with the same bits as the host fills.
    paged = P > 0 stores the caches in the paged layout with P-row blocks
    (keys "block_table", "block_rows", "paged_layout"); the logical cache
    contents are the same.  part = (e0, e1) keeps only the amateur and the
    contextual experts [e0, e1) of every query (contents as in the full
    workload; key "w" is the workload of the part)."""
    import torch
    stream = torch.cuda.current_stream() if stream is None else stream
    sp = stream.cuda_stream
    full = w
    if part is not None:
        w, seq_ids, cols = expert_part(full, *part)
        bl = base_lengths(full)[seq_ids]
    else:
        seq_ids, cols = np.arange(w.S, dtype=np.int32), slice(None)
        bl = base_lengths(w)
    lay = paged_layout(w, bl, paged, extra_steps) if paged else cache_layout(w, bl, extra_steps)
    k = torch.zeros(lay.total_elems, dtype=torch.bfloat16, device=device)
    v = torch.zeros(lay.total_elems, dtype=torch.bfloat16, device=device)
    cap = torch.from_numpy(lay.cap).to(device)
    base = torch.from_numpy(bl).to(device)
    ids = torch.from_numpy(seq_ids).to(device)
    extra = {}
    if paged:
        table = torch.from_numpy(lay.table).to(device)
        kv_off = torch.zeros(w.S, dtype=torch.int64, device=device)
        for tensor, buf in ((T_KCACHE, k), (T_VCACHE, v)):
            rc = dev_lib().synth_dev_fill_cache_paged(buf.data_ptr(), int(lay.layer_elems), table.data_ptr(),
                                                      lay.max_blocks, paged, base.data_ptr(), ids.data_ptr(), w.S,
                                                      w.L, w.Hkv, w.D, w.seed, tensor, normal_scale(SIGMA_KV), sp)
            if rc != 0:
                raise RuntimeError(f"synth_dev_fill_cache_paged failed: cuda error {rc}")
        extra = dict(block_table=table, block_rows=paged, paged_layout=lay)
    else:
        kv_off = torch.from_numpy(lay.kv_offset).to(device)
        dev_fill_caches(w, lay.layer_elems, k, v, kv_off, cap, base, ids, sp)
    emb = torch.empty((w.V, w.d), dtype=torch.bfloat16, device=device)
    wu = torch.empty((w.V, w.d), dtype=torch.bfloat16, device=device)
    dev_fill_matrix(w, T_EMBED, emb, sp)
    dev_fill_matrix(w, T_UNEMBED, wu, sp)
    # beta and r side by side in one allocation, so a per-step upload of both
    # can be one copy
    beta_r = torch.from_numpy(np.ascontiguousarray(np.stack([betas(full)[:, cols],
                                                             retrieval_scores(full)[:, cols]]))).to(device)
    return dict(k_cache=k, v_cache=v, kv_offset=kv_off, cap=cap, seq_len=base.clone(), base_len=bl, layout=lay,
                embed=emb, w_unembed=wu, beta=beta_r[0], r=beta_r[1], w=w, **extra)
