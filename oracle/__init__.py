"""CPU oracle of the PCED decode step (ctypes wrapper of pced_oracle.c).

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline / reference leg of ``bench.py``.  The decoding library
(``paper_2601_08670_gb300``) never imports, links or calls anything here.

The oracle computes, in fp64 and straight from the definitions, one decode
step of Parallel Context-of-Experts Decoding (paper Sec. 3): per-expert decode
attention over each expert's own cache, the unembedding with log-softmax, the
retrieval-aware contrastive score (Eq. 2) and the max over experts and tokens
(Eq. 3), with the chosen token appended to every expert's history.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIBDIR = os.path.join(HERE, "_lib")
RMS_EPS = 1e-6


def build(force: bool = False) -> str:
    os.makedirs(LIBDIR, exist_ok=True)
    so = os.path.join(LIBDIR, "liboracle_pced.so")
    srcs = [os.path.join(HERE, "pced_oracle.c"), os.path.join(HERE, "pced_oracle.h")]
    if force or not os.path.exists(so) or os.path.getmtime(so) < max(os.path.getmtime(p) for p in srcs):
        tmp = so + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math",
                               "-pthread", "-o", tmp, srcs[0], "-lm"])
        os.replace(tmp, so)
    return so


class _Dims(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("N", ctypes.c_int32), ("L", ctypes.c_int32), ("Hq", ctypes.c_int32),
                ("Hkv", ctypes.c_int32), ("D", ctypes.c_int32), ("V", ctypes.c_int32),
                ("gamma", ctypes.c_double), ("rms_eps", ctypes.c_double), ("attn_scale", ctypes.c_double),
                ("rope_theta", ctypes.c_double), ("score_mode", ctypes.c_int32), ("aggregation", ctypes.c_int32)]


_lib = None


def lib():
    global _lib
    if _lib is None:
        L = ctypes.CDLL(build())
        P, I32, I64, F64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_double
        L.oracle_bf16_value.argtypes = [ctypes.c_uint16]
        L.oracle_bf16_value.restype = F64
        L.oracle_round_bf16.argtypes = [F64]
        L.oracle_round_bf16.restype = ctypes.c_uint16
        L.oracle_rmsnorm.argtypes = [P, I32, F64, P]
        L.oracle_rmsnorm.restype = None
        L.oracle_attention.argtypes = [P, P, P, P, P, P, I32, I32, I32, I32, F64, P, I32]
        L.oracle_attention.restype = I32
        L.oracle_lm_head_logprobs.argtypes = [P, P, I32, I32, I32, P, P, I32]
        L.oracle_lm_head_logprobs.restype = I32
        L.oracle_contrastive_select.argtypes = [P, P, P, F64, I32, I32, I32, P, P, P, P, P]
        L.oracle_contrastive_select.restype = I32
        L.oracle_decode_step.argtypes = [ctypes.POINTER(_Dims), P, P, I64, P, P, P, P, P, P, P, P, P, P, P, P,
                                         P, P, I32]
        L.oracle_decode_step.restype = I32
        L.oracle_decode_step_ex.argtypes = list(L.oracle_decode_step.argtypes[:-1]) + [P, I32]
        L.oracle_decode_step_ex.restype = I32
        L.oracle_adacad_beta.argtypes = [P, I32, I32, I32, P]
        L.oracle_adacad_beta.restype = I32
        L.oracle_rope.argtypes = [P, I32, I64, F64, P]
        L.oracle_rope.restype = None
        L.oracle_relevance.argtypes = [P, I32, P, I32, F64, P]
        L.oracle_relevance.restype = I32
        L.oracle_aggregate_select.argtypes = [P, P, P, I32, I32, I32, I32, P, P, P, P]
        L.oracle_aggregate_select.restype = I32
        _lib = L
    return _lib


def threads() -> int:
    return max(1, min(256, os.cpu_count() or 1))


def _p(a: np.ndarray | None):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"], "oracle arrays must be C-contiguous"
    return a.ctypes.data


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def bf16_value(bits: int) -> float:
    return lib().oracle_bf16_value(int(bits))


def round_bf16(x: float) -> int:
    return int(lib().oracle_round_bf16(float(x)))


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact values of bf16 bit patterns (vectorised, for test convenience)."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def rmsnorm(x: np.ndarray, eps: float = RMS_EPS) -> np.ndarray:
    x = _c(x, np.float64)
    y = np.empty_like(x)
    lib().oracle_rmsnorm(_p(x), x.size, eps, _p(y))
    return y


def attention(q_bits, kc, vc, kv_off, cap, lens, Hq, Hkv, D, scale=None):
    """fp64 [S, Hq, D] decode-attention outputs of one layer."""
    q_bits = _c(q_bits, np.uint16)
    S = q_bits.shape[0]
    out = np.empty((S, Hq, D), dtype=np.float64)
    scale = 1.0 / math.sqrt(D) if scale is None else scale
    rc = lib().oracle_attention(_p(q_bits), _p(_c(kc, np.uint16)), _p(_c(vc, np.uint16)),
                                _p(_c(kv_off, np.int64)), _p(_c(cap, np.int32)), _p(_c(lens, np.int32)),
                                S, Hq, Hkv, D, scale, _p(out), threads())
    if rc != 0:
        raise ValueError(f"oracle_attention rc={rc}")
    return out


def lm_head_logprobs(h_bits, w_bits):
    h_bits = _c(h_bits, np.uint16)
    w_bits = _c(w_bits, np.uint16)
    S, d = h_bits.shape
    V = w_bits.shape[0]
    lp = np.empty((S, V), dtype=np.float64)
    lse = np.empty(S, dtype=np.float64)
    rc = lib().oracle_lm_head_logprobs(_p(h_bits), _p(w_bits), S, d, V, _p(lp), _p(lse), threads())
    if rc != 0:
        raise ValueError(f"oracle_lm_head_logprobs rc={rc}")
    return lp, lse


def contrastive_select(lp, beta, r, gamma, B, N):
    lp = _c(lp, np.float64)
    V = lp.shape[1]
    beta = _c(beta, np.float32)
    r = _c(r, np.float32)
    tok = np.empty(B, np.int32)
    exp_ = np.empty(B, np.int32)
    sc = np.empty(B, np.float64)
    tg = np.empty(B, np.float64)
    eg = np.empty(B, np.float64)
    rc = lib().oracle_contrastive_select(_p(lp), _p(beta), _p(r), float(gamma), B, N, V, _p(tok), _p(exp_),
                                         _p(sc), _p(tg), _p(eg))
    if rc != 0:
        raise ValueError(f"oracle_contrastive_select rc={rc}")
    return dict(token=tok, expert=exp_, score=sc, token_gap=tg, expert_gap=eg)


def rope(x, pos: int, theta: float) -> np.ndarray:
    """Rotary embedding of one head x [D] at position pos (rotate-half
    pairing, fp32 angles; see oracle_rope)."""
    x = _c(x, np.float64)
    y = np.empty_like(x)
    lib().oracle_rope(_p(x), x.size, int(pos), float(theta), _p(y))
    return y


def relevance(s, mode: int, z=None, eps: float = 1e-8) -> np.ndarray:
    """Relevance scores from raw retrieval scores s (mode 0 dense/ColBERT,
    1 sparse) and, if given, reranker logits z, fused by the harmonic mean
    (see oracle_relevance)."""
    s = _c(np.atleast_1d(s), np.float64)
    zz = None if z is None else _c(np.atleast_1d(z), np.float64)
    assert zz is None or zz.shape == s.shape
    r = np.empty_like(s)
    rc = lib().oracle_relevance(_p(s), int(mode), _p(zz), s.size, float(eps), _p(r))
    if rc != 0:
        raise ValueError(f"oracle_relevance rc={rc}")
    return r


MOE, POE = 1, 2


def aggregate_select(lp, beta, r, rule: int):
    """MoE (rule 1) / PoE (rule 2) aggregation of the contrastive expert
    distributions (see oracle_aggregate_select).  lp: [B*(N+1), V]; beta, r:
    [B, N].  Returns dict(token, expert, score, token_gap, expert_gap)."""
    lp = _c(lp, np.float64)
    beta = _c(beta, np.float32)
    r = _c(r, np.float32)
    B, N = beta.shape
    V = lp.shape[1]
    tok = np.empty(B, np.int32)
    ex = np.empty(B, np.int32)
    sc = np.empty(B, np.float64)
    gap = np.empty(B, np.float64)
    egap = np.empty(B, np.float64)
    rc = lib().oracle_aggregate_select(_p(lp), _p(beta), _p(r), B, N, V, int(rule), _p(tok), _p(ex), _p(sc), _p(gap),
                                       _p(egap))
    if rc != 0:
        raise ValueError(f"oracle_aggregate_select rc={rc}")
    return dict(token=tok, expert=ex, score=sc, token_gap=gap, expert_gap=egap)


def adacad_beta(lp, B, N):
    """Dynamic contrast strength (Sec. 3 after Eq. 2, as in AdaCAD): per
    expert, the Jensen-Shannon divergence in bits between its distribution
    exp(lp_k) and the amateur's exp(lp_0).  lp: [B*(N+1), V]; returns [B, N]."""
    lp = _c(lp, np.float64)
    V = lp.shape[1]
    out = np.empty((B, N), np.float64)
    rc = lib().oracle_adacad_beta(_p(lp), B, N, V, _p(out))
    if rc != 0:
        raise ValueError(f"oracle_adacad_beta rc={rc}")
    return out


def decode_step(dims: dict, kc, vc, layer_elems, kv_off, cap, lens, emb_rows, w_bits, beta, r,
                dynamic_beta: bool = False):
    """One full decode step; kc, vc and lens are updated in place.  With
    dynamic_beta the contrast strengths come from this step's distributions
    (adacad_beta, rounded to fp32; returned as "beta")."""
    dm = _Dims(dims["B"], dims["N"], dims["L"], dims["Hq"], dims["Hkv"], dims["D"], dims["V"],
               float(dims["gamma"]), float(dims.get("rms_eps", RMS_EPS)),
               float(dims.get("attn_scale", 1.0 / math.sqrt(dims["D"]))), float(dims.get("rope_theta", 0.0)),
               int(dims.get("score_mode", 0)), int(dims.get("aggregation", 0)))
    B, N = dims["B"], dims["N"]
    S, d = B * (N + 1), dims["Hq"] * dims["D"]
    for a, t in ((kc, np.uint16), (vc, np.uint16), (lens, np.int32)):
        assert a.dtype == t and a.flags["C_CONTIGUOUS"], "in-place arrays must be contiguous and typed"
    tok = np.empty(B, np.int32)
    exp_ = np.empty(B, np.int32)
    sc = np.empty(B, np.float64)
    tg = np.empty(B, np.float64)
    eg = np.empty(B, np.float64)
    h = np.empty((S, d), np.uint16)
    lse = np.empty(S, np.float64)
    bdyn = np.empty((B, N), np.float32) if dynamic_beta else None
    rc = lib().oracle_decode_step_ex(ctypes.byref(dm), _p(kc), _p(vc), int(layer_elems), _p(_c(kv_off, np.int64)),
                                     _p(_c(cap, np.int32)), _p(lens), _p(_c(emb_rows, np.uint16)),
                                     _p(_c(w_bits, np.uint16)), _p(_c(beta, np.float32)), _p(_c(r, np.float32)),
                                     _p(tok), _p(exp_), _p(sc), _p(tg), _p(eg), _p(h), _p(lse), _p(bdyn), threads())
    if rc != 0:
        raise ValueError(f"oracle_decode_step rc={rc}")
    out = dict(token=tok, expert=exp_, score=sc, token_gap=tg, expert_gap=eg, h=h, lse=lse)
    if dynamic_beta:
        out["beta"] = bdyn
    return out
