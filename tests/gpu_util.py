"""Helpers shared by the GPU parity tests: moving bf16 bit patterns between
numpy (oracle side) and torch device tensors (CUDA side)."""
import numpy as np
import torch


def to_dev_bf16(bits: np.ndarray, device="cuda") -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(device)


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def bits_to_f64(bits: np.ndarray) -> np.ndarray:
    return (np.asarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def near_tie(ref: dict, b: int, thr: float = 1e-3) -> bool:
    return ref["token_gap"][b] < thr or ref["expert_gap"][b] < thr
