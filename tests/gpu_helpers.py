"""Shared helpers of the GPU parity tests (device transfer and error metrics)."""
import numpy as np
import torch

from paper_2609_27373_gb300 import synth

# Tolerances for bf16 inputs with fp32 accumulation against the fp64 oracle.
O_MAX_ABS = 1e-2
O_REL_L2 = 5e-3
MASS_MAX_ABS = 1e-4     # per-step block mass r_qb
MASS_ROWSUM = 1e-5      # |sum_b r_qb - 1|


def to_dev(bits: np.ndarray) -> torch.Tensor:
    """uint16 bf16 bit patterns -> CUDA bf16 tensor (bit-identical)."""
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).cuda()


def bf16_dev_to_f64(t: torch.Tensor) -> np.ndarray:
    bits = t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    return synth.bf16_bits_to_f32(bits).astype(np.float64)


def empty_like_q(Q_bits: np.ndarray) -> torch.Tensor:
    return torch.empty(Q_bits.shape, dtype=torch.bfloat16, device="cuda")


def assert_close_o(got: np.ndarray, want: np.ndarray, what: str = "O"):
    err = np.abs(got - want)
    max_abs = float(err.max()) if err.size else 0.0
    denom = float(np.linalg.norm(want))
    rel = float(np.linalg.norm(got - want)) / denom if denom > 0 else float(np.linalg.norm(got))
    assert np.isfinite(got).all(), f"{what}: non-finite values"
    assert max_abs <= O_MAX_ABS, f"{what}: max-abs {max_abs:.3e} > {O_MAX_ABS}"
    assert rel <= O_REL_L2, f"{what}: rel-L2 {rel:.3e} > {O_REL_L2}"
    return max_abs, rel


def units_of(O_full: np.ndarray, units, block: int) -> np.ndarray:
    """Rows of the listed (b, h, q) query blocks, packed like the oracle's output."""
    return np.stack([O_full[b, h, q * block:(q + 1) * block] for b, h, q in units])


def sample_units(batch, n_heads, n_blocks, n, seed):
    """n (b, h, q) units including the first and last query blocks."""
    rng = np.random.default_rng(seed)
    units = {(0, 0, 0), (batch - 1, n_heads - 1, n_blocks - 1), (0, n_heads - 1, n_blocks // 2)}
    while len(units) < n:
        units.add((int(rng.integers(batch)), int(rng.integers(n_heads)), int(rng.integers(n_blocks))))
    return sorted(units)
