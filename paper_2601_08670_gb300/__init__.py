"""GB300 (sm_103a) decode step of Parallel Context-of-Experts Decoding.

Thin ctypes binding of ``libpced.so`` (C ABI declared in ``include/pced.h``):
argument marshalling only, every step of the computation runs in the
library's CUDA kernels.  PyTorch supplies device memory and streams.  There is
no CPU fallback: if the library is not built, every call raises.
"""
from __future__ import annotations

import ctypes
import math
import os

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
# PCED_LIB=checked selects the bounds-checked build (build.build(checked=True))
LIB_PATH = os.path.join(HERE, "_lib_checked" if os.environ.get("PCED_LIB") == "checked" else "_lib", "libpced.so")

PCED_DEV_BAD_LENGTH = 0x1
PCED_DEV_CACHE_FULL = 0x2
PCED_DEV_TIMEOUT = 0x4
PCED_DEV_BAD_TOKEN = 0x8
PCED_DEV_STEP_LIMIT = 0x10
PCED_DEV_BAD_BLOCK = 0x20
PCED_DEV_BOUNDS = 0x40


class PcedError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(msg)
        self.status = status


class Dims(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("N", ctypes.c_int32), ("L", ctypes.c_int32), ("Hq", ctypes.c_int32),
                ("Hkv", ctypes.c_int32), ("D", ctypes.c_int32), ("V", ctypes.c_int32)]


class StepArgs(ctypes.Structure):
    _fields_ = [("dims", Dims), ("embed", ctypes.c_void_p), ("w_unembed", ctypes.c_void_p),
                ("k_cache", ctypes.c_void_p), ("v_cache", ctypes.c_void_p), ("layer_elems", ctypes.c_int64),
                ("kv_offset", ctypes.c_void_p), ("cap", ctypes.c_void_p), ("total_cap", ctypes.c_int64),
                ("seq_len", ctypes.c_void_p), ("step", ctypes.c_void_p), ("history", ctypes.c_void_p),
                ("expert_trace", ctypes.c_void_p), ("score_trace", ctypes.c_void_p), ("gap_trace", ctypes.c_void_p),
                ("max_steps", ctypes.c_int32),
                ("beta", ctypes.c_void_p), ("r", ctypes.c_void_p), ("gamma", ctypes.c_float),
                ("attn_scale", ctypes.c_float), ("rms_eps", ctypes.c_float), ("bos_token", ctypes.c_int32),
                ("hidden_out", ctypes.c_void_p), ("lse_out", ctypes.c_void_p), ("workspace", ctypes.c_void_p),
                ("workspace_bytes", ctypes.c_size_t), ("stage_events", ctypes.c_void_p),
                ("n_stage_events", ctypes.c_int32), ("beta_from_step", ctypes.c_int32), ("beta_out", ctypes.c_void_p),
                ("block_table", ctypes.c_void_p), ("block_rows", ctypes.c_int32), ("max_blocks", ctypes.c_int32),
                ("rope_theta", ctypes.c_float), ("score_mode", ctypes.c_int32), ("aggregation", ctypes.c_int32),
                ("wait_limit_ns", ctypes.c_uint64), ("expert_base", ctypes.c_int32), ("key_out", ctypes.c_void_p),
                ("token_out", ctypes.c_void_p), ("expert_out", ctypes.c_void_p), ("score_out", ctypes.c_void_p)]


_lib = None


def lib(path: str = LIB_PATH):
    """Load libpced.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is missing: build it with paper_2601_08670_gb300.build.build()")
        L = ctypes.CDLL(path)
        P, I32, I64, SZ, F = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t, ctypes.c_float
        L.pced_status_string.argtypes = [I32]
        L.pced_status_string.restype = ctypes.c_char_p
        L.pced_last_error.argtypes = []
        L.pced_last_error.restype = ctypes.c_char_p
        L.pced_decode_attention_workspace_size.argtypes = [I32, I32, I32, I32]
        L.pced_decode_attention_workspace_size.restype = SZ
        L.pced_decode_attention.argtypes = [P, P, P, I64, P, P, P, I32, I32, I32, I32, I64, F, P, P, SZ, P]
        L.pced_decode_attention.restype = I32
        L.pced_decode_attention_noalloc.argtypes = [P, P, P, I64, P, P, P, I32, I32, I32, I32, I64, F, P, P, P]
        L.pced_decode_attention_noalloc.restype = I32
        L.pced_lm_head_workspace_size.argtypes = [I32, I32]
        L.pced_lm_head_workspace_size.restype = SZ
        L.pced_lm_head_logprobs.argtypes = [P, P, I32, I32, I32, P, P, P, SZ, P]
        L.pced_lm_head_logprobs.restype = I32
        L.pced_contrastive_select_workspace_size.argtypes = [I32, I32, I32]
        L.pced_contrastive_select_workspace_size.restype = SZ
        L.pced_contrastive_select.argtypes = [P, P, P, F, I32, I32, I32, P, P, P, P, SZ, P]
        L.pced_contrastive_select.restype = I32
        L.pced_adacad_beta_workspace_size.argtypes = [I32, I32, I32]
        L.pced_adacad_beta_workspace_size.restype = SZ
        L.pced_adacad_beta.argtypes = [P, I32, I32, I32, P, P, SZ, P]
        L.pced_adacad_beta.restype = I32
        L.pced_relevance.argtypes = [P, I32, P, I32, ctypes.c_double, P, P]
        L.pced_relevance.restype = I32
        L.pced_step_workspace_size.argtypes = [ctypes.POINTER(Dims)]
        L.pced_step_workspace_size.restype = SZ
        L.pced_step.argtypes = [ctypes.POINTER(StepArgs), P]
        L.pced_step.restype = I32
        L.pced_step_host_io.argtypes = [ctypes.POINTER(StepArgs), P, P, P, P, P, P]
        L.pced_step_host_io.restype = I32
        L.pced_step_launch_count.argtypes = [ctypes.POINTER(StepArgs)]
        L.pced_step_launch_count.restype = I32
        L.pced_step_launch_kind.argtypes = [ctypes.POINTER(StepArgs), I32]
        L.pced_step_launch_kind.restype = ctypes.c_char_p
        L.pced_select_key.argtypes = [F, I32, I32]
        L.pced_select_key.restype = I64
        L.pced_select_key_unpack.argtypes = [I64, ctypes.POINTER(F), ctypes.POINTER(I32), ctypes.POINTER(I32)]
        L.pced_select_key_unpack.restype = None
        L.pced_step_commit.argtypes = [P, I32, P, P, P, P, I32, P, P]
        L.pced_step_commit.restype = I32
        _lib = L
    return _lib


def _check(rc: int, what: str):
    if rc != 0:
        L = lib()
        raise PcedError(rc, f"{what}: {L.pced_status_string(rc).decode()}: {L.pced_last_error().decode()}")


def _require(cond: bool, what: str):
    """Argument check of the binding (raises even under python -O)."""
    if not cond:
        raise ValueError(what)


def _ptr(t):
    return None if t is None else t.data_ptr()


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


def workspace(nbytes: int, device) -> torch.Tensor:
    """Zeroed workspace (the device status word at byte 0 starts clear)."""
    return torch.zeros(max(int(nbytes), 256), dtype=torch.uint8, device=device)


def device_status(ws: torch.Tensor) -> int:
    """Device status bits the kernels ORed into the workspace (synchronises)."""
    return int(ws[:4].view(torch.int32).item())


# ------------------------------------------------------------------ entry points
def decode_attention_workspace_size(S, Hq, Hkv, D) -> int:
    return int(lib().pced_decode_attention_workspace_size(S, Hq, Hkv, D))


def decode_attention(q, k_cache, v_cache, kv_offset, cap, seq_len, Hkv: int, total_cap: int, scale=None, out=None,
                     ws=None, stream=None):
    """pced_decode_attention: q bf16 [S, Hq, D]; caches bf16 (one layer); returns fp32 [S, Hq, D]."""
    S, Hq, D = q.shape
    scale = 1.0 / math.sqrt(D) if scale is None else scale
    if out is None:
        out = torch.empty((S, Hq, D), dtype=torch.float32, device=q.device)
    if ws is None:
        ws = workspace(decode_attention_workspace_size(S, Hq, Hkv, D), q.device)
    _check(lib().pced_decode_attention(_ptr(q), _ptr(k_cache), _ptr(v_cache), k_cache.numel(), _ptr(kv_offset),
                                       _ptr(cap), _ptr(seq_len), S, Hq, Hkv, D, int(total_cap), float(scale),
                                       _ptr(out), _ptr(ws), ws.numel(), _stream(stream)), "pced_decode_attention")
    return out


# fixed size of the library's scratch array behind decode_attention_noalloc
NOALLOC_SCRATCH_BYTES = 16 << 20


def decode_attention_noalloc(q, k_cache, v_cache, kv_offset, cap, seq_len, Hkv: int, total_cap: int, out,
                             scale=None, status=None, stream=None):
    """pced_decode_attention_noalloc: decode_attention without a workspace.

    For callers that cannot allocate device memory when they run attention
    (allocator locked or shutting down, host callbacks, capped memory pools):
    the partial records live in a fixed library-owned device array, so the
    caller passes the output buffer ``out`` (fp32 [S, Hq, D]) and, optionally,
    an int32 device ``status`` word.  Calls share that array: overlapping calls
    on the GPU race.  The first call on a device should come before any stream
    capture on it."""
    S, Hq, D = q.shape
    scale = 1.0 / math.sqrt(D) if scale is None else scale
    _check(lib().pced_decode_attention_noalloc(_ptr(q), _ptr(k_cache), _ptr(v_cache), k_cache.numel(),
                                               _ptr(kv_offset), _ptr(cap), _ptr(seq_len), S, Hq, Hkv, D,
                                               int(total_cap), float(scale), _ptr(out),
                                               None if status is None else _ptr(status), _stream(stream)),
           "pced_decode_attention_noalloc")
    return out


def lm_head_workspace_size(S, V) -> int:
    return int(lib().pced_lm_head_workspace_size(S, V))


def lm_head_logprobs(hidden, w_unembed, logprobs=None, lse=None, ws=None, stream=None):
    """pced_lm_head_logprobs: hidden bf16 [S, d], W bf16 [V, d] -> (fp32 [S, V], fp32 [S])."""
    S, d = hidden.shape
    V = w_unembed.shape[0]
    if logprobs is None:
        logprobs = torch.empty((S, V), dtype=torch.float32, device=hidden.device)
    if lse is None:
        lse = torch.empty(S, dtype=torch.float32, device=hidden.device)
    if ws is None:
        ws = workspace(lm_head_workspace_size(S, V), hidden.device)
    _check(lib().pced_lm_head_logprobs(_ptr(hidden), _ptr(w_unembed), S, d, V, _ptr(logprobs), _ptr(lse), _ptr(ws),
                                       ws.numel(), _stream(stream)), "pced_lm_head_logprobs")
    return logprobs, lse


def contrastive_select_workspace_size(B, N, V) -> int:
    return int(lib().pced_contrastive_select_workspace_size(B, N, V))


def contrastive_select(logprobs, beta, r, gamma: float, ws=None, stream=None):
    """pced_contrastive_select: returns (token [B] int32, expert [B] int32, score [B] fp32)."""
    B, N = beta.shape
    V = logprobs.shape[1]
    dev = logprobs.device
    token = torch.empty(B, dtype=torch.int32, device=dev)
    expert = torch.empty(B, dtype=torch.int32, device=dev)
    score = torch.empty(B, dtype=torch.float32, device=dev)
    if ws is None:
        ws = workspace(contrastive_select_workspace_size(B, N, V), dev)
    _check(lib().pced_contrastive_select(_ptr(logprobs), _ptr(beta), _ptr(r), float(gamma), B, N, V, _ptr(token),
                                         _ptr(expert), _ptr(score), _ptr(ws), ws.numel(), _stream(stream)),
           "pced_contrastive_select")
    return token, expert, score


def adacad_beta(logprobs, B: int, N: int, ws=None, stream=None):
    """pced_adacad_beta: per-expert Jensen-Shannon divergence (bits) between
    each expert's distribution and its query's amateur, fp32 [B, N]."""
    V = logprobs.shape[1]
    beta = torch.empty((B, N), dtype=torch.float32, device=logprobs.device)
    if ws is None:
        ws = workspace(int(lib().pced_adacad_beta_workspace_size(B, N, V)), logprobs.device)
    _check(lib().pced_adacad_beta(_ptr(logprobs), B, N, V, _ptr(beta), _ptr(ws), ws.numel(), _stream(stream)),
           "pced_adacad_beta")
    return beta


RET_DENSE, RET_SPARSE = 0, 1
SCORE_LOGPROB, SCORE_LOGIT = 0, 1
AGG_MAX, AGG_MOE, AGG_POE = 0, 1, 2


def relevance(ret_scores, ret_mode: int = RET_DENSE, rer_logits=None, eps: float = 1e-8, stream=None):
    """pced_relevance: relevance scores in [0, 1) from raw retrieval scores
    (dense/ColBERT or sparse) and optional reranker logits, fused by the
    harmonic mean (fp32 tensors of one shape on the device)."""
    _require(ret_scores.dtype == torch.float32 and ret_scores.is_contiguous(), "ret_scores: contiguous fp32")
    if rer_logits is not None:
        _require(rer_logits.dtype == torch.float32 and rer_logits.is_contiguous(), "rer_logits: contiguous fp32")
        _require(rer_logits.shape == ret_scores.shape, "rer_logits: the shape of ret_scores")
    r = torch.empty_like(ret_scores)
    _check(lib().pced_relevance(_ptr(ret_scores), int(ret_mode), _ptr(rer_logits), ret_scores.numel(), float(eps),
                                _ptr(r), _stream(stream)), "pced_relevance")
    return r


def dims(B, N, L, Hq, Hkv, D, V) -> Dims:
    return Dims(B, N, L, Hq, Hkv, D, V)


def step_workspace_size(dm: Dims) -> int:
    return int(lib().pced_step_workspace_size(ctypes.byref(dm)))


def step_launch_count(args) -> int:
    """Kernel launches of one pced_step call with these StepArgs."""
    return int(lib().pced_step_launch_count(ctypes.byref(args)))


def select_key(score: float, token: int, expert: int) -> int:
    """Eq. 3's choice as an int64 whose signed order is Eq. 3's order
    (pced_select_key)."""
    return int(lib().pced_select_key(float(score), int(token), int(expert)))


def select_key_unpack(key: int):
    """(fp32 score, token, expert) of a packed key."""
    s, t, e = ctypes.c_float(), ctypes.c_int32(), ctypes.c_int32()
    lib().pced_select_key_unpack(int(key), ctypes.byref(s), ctypes.byref(t), ctypes.byref(e))
    return s.value, t.value, e.value


def step_launch_kinds(args) -> list:
    return [lib().pced_step_launch_kind(ctypes.byref(args), i).decode() for i in range(step_launch_count(args))]


class Decoder:
    """Device-resident PCED decoding state and the pced_step call.

    Holds references to the caller's caches and weights, and owns the step
    counter, the generated history, the expert trace and the workspace.  Each
    ``step()`` is one pced_step call (asynchronous on the current stream)."""

    def __init__(self, dm: Dims, *, embed, w_unembed, k_cache, v_cache, layer_elems: int, kv_offset, cap, seq_len,
                 beta, r, gamma: float, max_steps: int, total_cap: int, bos: int = 0, attn_scale=None,
                 rms_eps: float = 1e-6, keep_hidden: bool = False, dynamic_beta: bool = False, block_table=None,
                 block_rows: int = 0, rope_theta: float = 0.0, score_mode: int = 0, aggregation: int = 0,
                 track_gaps: bool = True):
        dev = k_cache.device
        self.dm = dm
        B, S, d = dm.B, dm.B * (dm.N + 1), dm.Hq * dm.D
        self.step_t = torch.zeros(1, dtype=torch.int32, device=dev)
        self.history = torch.zeros((B, max_steps), dtype=torch.int32, device=dev)
        self.expert_trace = torch.zeros((B, max_steps), dtype=torch.int32, device=dev)
        self.score_trace = torch.zeros((B, max_steps), dtype=torch.float32, device=dev)
        # near-tie margins of every choice: [B, max_steps, 2] (token gap, expert gap)
        self.gap_trace = torch.zeros((B, max_steps, 2), dtype=torch.float32, device=dev) if track_gaps else None
        # this step's choice at fixed addresses (the traces move with t)
        # (one [3, B] block, so that reading all three back is one copy)
        self._choice = torch.zeros((3, B), dtype=torch.int32, device=dev)
        self.token_out, self.expert_out = self._choice[0], self._choice[1]
        self.score_out = self._choice[2].view(torch.float32)
        self.hidden = torch.zeros((S, d), dtype=torch.bfloat16, device=dev) if keep_hidden else None
        self.lse = torch.zeros(S, dtype=torch.float32, device=dev)
        self.ws = workspace(step_workspace_size(dm), dev)
        self._keep = (embed, w_unembed, k_cache, v_cache, kv_offset, cap, seq_len, beta, r, block_table)
        self.seq_len = seq_len
        self.beta, self.r = beta, r
        self.args = StepArgs(
            dm, _ptr(embed), _ptr(w_unembed), _ptr(k_cache), _ptr(v_cache), int(layer_elems), _ptr(kv_offset),
            _ptr(cap), int(total_cap), _ptr(seq_len), _ptr(self.step_t), _ptr(self.history),
            _ptr(self.expert_trace), _ptr(self.score_trace), _ptr(self.gap_trace), int(max_steps), _ptr(beta), _ptr(r),
            float(gamma),
            float(1.0 / math.sqrt(dm.D) if attn_scale is None else attn_scale), float(rms_eps), int(bos),
            _ptr(self.hidden), _ptr(self.lse), _ptr(self.ws), self.ws.numel())
        self.max_steps = max_steps
        self.args.token_out = _ptr(self.token_out)
        self.args.expert_out = _ptr(self.expert_out)
        self.args.score_out = _ptr(self.score_out)
        self.args.rope_theta = float(rope_theta)  # rotary base, 0: none
        self.args.score_mode = int(score_mode)     # SCORE_LOGPROB / SCORE_LOGIT
        self.args.aggregation = int(aggregation)   # AGG_MAX / AGG_MOE / AGG_POE
        if block_table is not None:  # paged caches
            _require(block_table.dtype == torch.int32 and block_table.is_contiguous() and block_table.dim() == 2,
                     "block_table: contiguous int32 [S, max_blocks]")
            self.args.block_table = _ptr(block_table)
            self.args.block_rows = int(block_rows)
            self.args.max_blocks = int(block_table.shape[1])
        # dynamic contrast strength: the first step computes beta (into the
        # `beta` tensor, which the later steps read) from its distributions
        if dynamic_beta:
            _require(beta.dtype == torch.float32 and beta.is_contiguous(),
                     "beta: contiguous fp32 (dynamic beta writes it)")
            self.args.beta_from_step = 1
            self.args.beta_out = _ptr(beta)

    def step(self, stream=None):
        _check(lib().pced_step(ctypes.byref(self.args), _stream(stream)), "pced_step")
        self.args.beta_from_step = 0

    def step_host_io(self, beta=None, r=None, token=None, expert=None, score=None, stream=None):
        """One step with host buffers (pced_step_host_io): uploads `beta` / `r`
        (host fp32 [B, N], None: keep the device values), steps, and copies
        the choice into `token` / `expert` / `score` (host [B] int32 / int32 /
        fp32, None: skip).  Asynchronous on the stream; use page-locked
        tensors (pin_memory()) for asynchronous copies and graph capture.
        Adjacent buffers on both sides (r right after beta; expert after
        token, score after expert, as choice_buffers() lays them out) move
        in one copy each way."""
        B, N = self.dm.B, self.dm.N

        def host(t, dtype, n):
            if t is None:
                return None
            _require(t.device.type == "cpu" and t.dtype == dtype and t.is_contiguous() and t.numel() == n,
                     f"host buffers: contiguous {dtype} CPU tensors of {n} elements")
            return t.data_ptr()

        _check(lib().pced_step_host_io(ctypes.byref(self.args), host(beta, torch.float32, B * N),
                                       host(r, torch.float32, B * N), host(token, torch.int32, B),
                                       host(expert, torch.int32, B), host(score, torch.float32, B),
                                       _stream(stream)), "pced_step_host_io")
        self.args.beta_from_step = 0

    def choice_buffers(self):
        """Page-locked host (token, expert, score) tensors laid out like the
        device outputs, so step_host_io reads them back in one copy."""
        blk = torch.zeros((3, self.dm.B), dtype=torch.int32).pin_memory()
        return blk[0], blk[1], blk[2].view(torch.float32)

    def capture_host_io(self, beta=None, r=None, token=None, expert=None, score=None):
        """A CUDA graph of one step_host_io call: each replay is one decode
        step with its uploads and read-backs (page-locked host tensors
        required; the decoder's dynamic-beta first step must already be done)."""
        _require(not self.args.beta_from_step, "run the dynamic-beta first step before capturing")
        for t in (beta, r, token, expert, score):
            _require(t is None or t.is_pinned(), "graph capture needs page-locked host tensors")
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            self.step_host_io(beta, r, token, expert, score)
        return g

    def step_partial(self, keys, expert_base: int, stream=None):
        """Expert-partitioned step: this decoder's experts are global experts
        expert_base + 1 .. expert_base + N; writes their best choice per query
        as packed keys (int64 [B] device tensor `keys`) and appends nothing.
        Reduce the keys with a max over the decoders (NCCL / gloo all-reduce,
        torch.maximum), then call commit()."""
        _require(keys.dtype == torch.int64 and keys.is_contiguous() and keys.numel() >= self.dm.B,
                 "keys: contiguous int64 of at least B elements")
        self.args.key_out = _ptr(keys)
        self.args.expert_base = int(expert_base)
        try:
            self.step(stream)
        finally:
            self.args.key_out = None
            self.args.expert_base = 0

    def commit(self, keys, stream=None):
        """Append the reduced choices (int64 [B] device keys) and advance t."""
        _check(lib().pced_step_commit(_ptr(keys), self.dm.B, _ptr(self.step_t), _ptr(self.history),
                                      _ptr(self.expert_trace), _ptr(self.score_trace), self.max_steps,
                                      _ptr(self.ws), _stream(stream)), "pced_step_commit")

    def set_stage_events(self, events):
        """Record one torch.cuda.Event before and after every launch of each
        subsequent step (None disables)."""
        if events is None:
            self._events = None
            self.args.stage_events = None
            self.args.n_stage_events = 0
            return
        for ev in events:  # torch creates the CUDA event on its first record
            if ev.cuda_event == 0:
                ev.record()
        torch.cuda.synchronize()
        self._events = events
        self._event_handles = (ctypes.c_void_p * len(events))(*[ev.cuda_event for ev in events])
        self.args.stage_events = ctypes.cast(self._event_handles, ctypes.c_void_p)
        self.args.n_stage_events = len(events)

    def launches_per_step(self) -> int:
        """Kernel launches of the next step() call."""
        return step_launch_count(self.args)

    def launch_kinds(self) -> list:
        return step_launch_kinds(self.args)

    def status(self) -> int:
        return device_status(self.ws)


def decoder_from_inputs(dm: Dims, t: dict, *, gamma: float, max_steps: int, bos: int = 0, keep_hidden=False,
                        attn_scale=None, rms_eps: float = 1e-6, dynamic_beta: bool = False,
                        rope_theta: float = 0.0, score_mode: int = 0, aggregation: int = 0,
                        track_gaps: bool = True) -> Decoder:
    """Decoder over a dict of device tensors with the keys k_cache, v_cache,
    kv_offset, cap, seq_len, embed, w_unembed, beta, r, and the host layout
    values layer_elems / total_cap (or a `layout` object carrying them)."""
    lay = t.get("layout")
    layer_elems = t["layer_elems"] if "layer_elems" in t else lay.layer_elems
    total_cap = t["total_cap"] if "total_cap" in t else int(lay.cap.astype("int64").sum())
    return Decoder(dm, embed=t["embed"], w_unembed=t["w_unembed"], k_cache=t["k_cache"], v_cache=t["v_cache"],
                   layer_elems=layer_elems, kv_offset=t["kv_offset"], cap=t["cap"], seq_len=t["seq_len"],
                   beta=t["beta"], r=t["r"], gamma=gamma, max_steps=max_steps, total_cap=total_cap, bos=bos,
                   attn_scale=attn_scale, rms_eps=rms_eps, keep_hidden=keep_hidden, dynamic_beta=dynamic_beta,
                   block_table=t.get("block_table"), block_rows=int(t.get("block_rows", 0)), rope_theta=rope_theta,
                   score_mode=score_mode, aggregation=aggregation, track_gaps=track_gaps)
