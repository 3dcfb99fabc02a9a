"""Seeded synthetic inputs shared by the tests, the smoke check and the bench.

This module draws random numbers and nothing else: it holds none of the DQT
arithmetic (no quantiser, no GEMM, no optimiser, no rounding), so that the CUDA
path and the CPU oracle, which must share no code, can both be fed the very
same bytes.  All draws use a CPU ``torch.Generator`` so that the bytes do not
depend on the device.

Value distributions follow the LLaMA-shaped workloads the paper trains
(Sec. 4.1): activations ~ N(0, 1) in bf16, upstream gradients ~ N(0, 1e-2) in
bf16 (1e-2 read as the standard deviation), dense initial weights
~ N(0, 0.02) in fp32 (the usual LLaMA initialiser), optimiser moments zero.
"""
import torch

__all__ = ["normal", "bf16_bits", "uniform_u32"]


def normal(shape, std: float, seed: int, dtype=torch.float32) -> torch.Tensor:
    """N(0, std^2) draws from a CPU generator seeded with ``seed``, cast to ``dtype``."""
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    x = torch.randn(*shape, generator=g, dtype=torch.float32)
    if std != 1.0:
        x.mul_(std)
    return x.to(dtype)


def uniform_u32(n: int, seed: int) -> torch.Tensor:
    """n uniform 32-bit words (as int64 holding the unsigned value)."""
    g = torch.Generator(device="cpu")
    g.manual_seed(int(seed))
    return torch.randint(0, 2**32, (n,), generator=g, dtype=torch.int64)


def bf16_bits(t: torch.Tensor):
    """Raw bits of a CPU bf16 tensor as a numpy uint16 array (no arithmetic)."""
    assert t.dtype == torch.bfloat16 and t.device.type == "cpu"
    return t.contiguous().view(torch.int16).numpy().view("uint16")
