"""The paper's roofline and energy model of a spiking linear layer (Sec. IV-A and IV-B,
Eq. (12)-(16), Table I), evaluated on measured spike sparsities.

Host arithmetic only (no kernel): the CUDA path measures, per spiking-linear launch, the
spikes of its input block and the rows of W^T it had to fetch; this module turns them
into the per-token operation and data loads of Eq. (12)-(13), the token latency of
Eq. (14) on a platform with L_ops operations/s and L_data bits/s, the end-to-end token
throughput of Eq. (15) (encoder linears once per token, decoder linears once per
denoising step) and the energy per token of Eq. (16).

Readings (the paper's text garbles two of them):
- a linear of d_in inputs and d_out outputs generalises Eq. (12)-(13)'s D x D layer:
  N_ops = 2 T d_in d_out (1 - sigma) and N_data = d_in d_out (1 - sigma^{BT}) b_W / B;
- the memory-bound branch of Eq. (14) is N_data / L_data (N_data is already per token);
- the decoder term of Eq. (15)-(16) sums over the decoder's layers and steps.
"""
from dataclasses import dataclass
from typing import Iterable, List, Optional


@dataclass(frozen=True)
class Platform:
    name: str
    l_ops: float   # operations per second
    l_data: float  # bits per second
    e_ops: float   # joules per operation
    e_data: float  # joules per bit


# Table I of the paper (context only: these are the paper's modelled systems).
OCMS = Platform("OCMS (paper Table I)", 300e12, 8e12, 0.05e-12, 10e-12)
ICMS = Platform("ICMS (paper Table I)", 20e12, 30e12, 0.05e-12, 0.5e-12)


def gb300(bf16_tflops, hbm_gbs, name="GB300 (measured)"):
    """This GPU as an Eq. (14) platform: the measured dense bf16 tensor rate as L_ops and
    the measured HBM copy bandwidth (bytes/s x 8) as L_data; no energy figures."""
    return Platform(name, bf16_tflops * 1e12, hbm_gbs * 1e9 * 8.0, 0.0, 0.0)


@dataclass(frozen=True)
class Linear:
    """One linear of the model as it runs on a block: its shape, the block, the measured
    input sparsity sigma = P(x = 0) (Sec. IV-A) and where it runs."""
    d_in: int
    d_out: int
    B: int
    T: int
    sigma: float
    part: str = "dec"         # "enc": once per block (context pass); "dec": once per step
    rows_frac: Optional[float] = None  # measured fraction of W^T rows fetched, if known


def n_ops(l: Linear) -> float:
    """Eq. (12): operations per token, 2 T d_in d_out (1 - sigma)."""
    return 2.0 * l.T * l.d_in * l.d_out * (1.0 - l.sigma)


def n_data(l: Linear, b_w: float, measured_rows: bool = False) -> float:
    """Eq. (13): bits fetched per token, d_in d_out (1 - sigma^{BT}) b_W / B; with
    measured_rows the i.i.d. fraction 1 - sigma^{BT} is replaced by the measured one."""
    frac = l.rows_frac if (measured_rows and l.rows_frac is not None) else \
        1.0 - l.sigma ** (l.B * l.T)
    return l.d_in * l.d_out * frac * b_w / l.B


def token_latency(l: Linear, p: Platform, b_w: float, measured_rows: bool = False) -> float:
    """Eq. (14): max(N_ops / L_ops, N_data / L_data), seconds per token."""
    return max(n_ops(l) / p.l_ops, n_data(l, b_w, measured_rows) / p.l_data)


def bound(l: Linear, p: Platform, b_w: float) -> str:
    return "compute" if n_ops(l) / p.l_ops >= n_data(l, b_w) / p.l_data else "memory"


def e2e_throughput(linears: Iterable[Linear], p: Platform, b_w: float, S: int,
                   measured_rows: bool = False) -> float:
    """Eq. (15): tokens/s = 1 / (sum over encoder linears of TL + sum over decoder
    linears and the S denoising steps of TL).  A decoder linear listed once stands for
    the same linear at every step."""
    total = 0.0
    for l in linears:
        tl = token_latency(l, p, b_w, measured_rows)
        total += tl if l.part == "enc" else S * tl
    return 1.0 / total if total > 0 else float("inf")


def energy_per_token(linears: Iterable[Linear], p: Platform, b_w: float, S: int,
                     measured_rows: bool = False) -> float:
    """Eq. (16): joules per token, sum of N_ops E_ops + N_data E_data (decoder x S)."""
    e = 0.0
    for l in linears:
        x = n_ops(l) * p.e_ops + n_data(l, b_w, measured_rows) * p.e_data
        e += x if l.part == "enc" else S * x
    return e


def dense(linears: List[Linear]) -> List[Linear]:
    """The same model without spike sparsity (an MDLM, sigma = 0)."""
    return [Linear(l.d_in, l.d_out, l.B, l.T, 0.0, l.part, 1.0) for l in linears]


def autoregressive(linears: List[Linear]) -> List[Linear]:
    """The AR special case: one token per block (B = 1), sigma = 0 (Sec. IV-A)."""
    return [Linear(l.d_in, l.d_out, 1, l.T, 0.0, l.part, 1.0) for l in linears]
