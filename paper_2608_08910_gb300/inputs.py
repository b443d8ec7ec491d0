"""Seeded synthetic inputs shaped like the paper's MoE expert workload.

This module only draws random numbers: it holds none of the tq2_0_fx4
arithmetic, and both the CUDA path and the CPU oracle take their inputs from
it. The paper's real weights (DeepSeek-V4-Flash routed experts, 256 experts
of 4096 x 2048 per projection) are not available; these generators stand in
for them with the same shapes:

  - expert weights: Student-t(nu = 5) * 0.02 (heavy-tailed, like trained
    weights), drawn as z / sqrt(chi2_5 / 5), one generator per
    (seed, expert, projection) so any single expert can be regenerated alone;
  - the 1024 x 1024 single-GEMV matrix: N(0, 0.02);
  - router weights: N(0, 0.02) [n_experts][hidden];
  - hidden states: N(0, 1);
  - the skewed-routing bias: -s * ln(rank), rank = expert index + 1
    (a Zipf(s) prior on expert popularity);
  - trit planes: independent uniform draws from {-1, 0, 1} with f16 scales
    |N(0, 0.01)|.
"""
import torch

PROJ_GATE, PROJ_UP, PROJ_DOWN = 0, 1, 2


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=torch.device(device))
    g.manual_seed(int(seed) & ((1 << 63) - 1))
    return g


def normal(shape, std: float, seed: int, device="cpu") -> torch.Tensor:
    g = _gen(seed, device)
    return torch.randn(shape, generator=g, device=device, dtype=torch.float32) * std


def student_t(shape, nu: int, scale: float, seed: int, device="cpu") -> torch.Tensor:
    g = _gen(seed, device)
    z = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
    chi2 = torch.zeros(shape, device=device, dtype=torch.float32)
    for _ in range(nu):
        e = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
        chi2.add_(e * e)
    return z / torch.sqrt(chi2 / nu) * scale


def expert_seed(seed: int, expert: int, proj: int) -> int:
    return (int(seed) << 24) + 3 * int(expert) + int(proj) + 1


def expert_matrix(seed: int, expert: int, proj: int, hidden: int, inter: int,
                  device="cpu") -> torch.Tensor:
    """fp32 weight of one expert projection: gate/up are [inter][hidden],
    down is [hidden][inter]."""
    shape = (hidden, inter) if proj == PROJ_DOWN else (inter, hidden)
    return student_t(shape, 5, 0.02, expert_seed(seed, expert, proj), device)


def gemv_matrix(seed: int, n: int, k: int, device="cpu") -> torch.Tensor:
    return normal((n, k), 0.02, (int(seed) << 24) + 7, device)


def router_weight(seed: int, n_experts: int, hidden: int, device="cpu") -> torch.Tensor:
    return normal((n_experts, hidden), 0.02, (int(seed) << 24) + 11, device)


def hidden_states(seed: int, tokens: int, hidden: int, device="cpu", stream: int = 0) -> torch.Tensor:
    return normal((tokens, hidden), 1.0, (int(seed) << 24) + 13 + (int(stream) << 8), device)


def zipf_bias(n_experts: int, s: float = 1.1) -> torch.Tensor:
    ranks = torch.arange(1, n_experts + 1, dtype=torch.float64)
    return (-s * torch.log(ranks)).to(torch.float32)


def trit_planes(seed: int, n: int, k: int, device="cpu"):
    """t1, t2 int8 [n][k] uniform on {-1, 0, 1}; f16 scales [n][k/256]."""
    g = _gen((int(seed) << 24) + 17, device)
    t1 = torch.randint(-1, 2, (n, k), generator=g, device=device, dtype=torch.int8)
    t2 = torch.randint(-1, 2, (n, k), generator=g, device=device, dtype=torch.int8)
    s = torch.randn((n, max(k // 256, 0)), generator=g, device=device).abs() * 0.01
    return t1, t2, s.to(torch.float16)


def log_uniform_scale_matrix(seed: int, n: int, k: int, device="cpu") -> torch.Tensor:
    """N(0,1) weights with a per-(row, 256-block) scale spread over eight
    decades, so one matrix exercises tiny, normal and large f16 scales."""
    g = _gen((int(seed) << 24) + 19, device)
    w = torch.randn((n, k), generator=g, device=device)
    e = torch.rand((n, max(k // 256, 1)), generator=g, device=device) * 8.0 - 6.0
    sc = torch.pow(10.0, e).repeat_interleave(256, dim=1)[:, :k]
    return (w * sc).to(torch.float32)


def mxfp4_matrix(seed: int, n: int, k: int, device="cpu") -> torch.Tensor:
    """Random MXFP4 bytes for an n x k matrix (17 bytes per 32 elements: an
    e8m0 scale byte, then 16 bytes of e2m1 nibbles), standing in for released
    MXFP4 expert weights: scale bytes 119..124 (2^-8 .. 2^-3), magnitude codes
    drawn with weights falling from 0 to 7 as in quantized heavy-tailed
    weights, random signs. Random bytes only: no quantizer runs here."""
    g = _gen((int(seed) << 24) + 23, device)
    nb = n * (k // 32)
    scale = torch.randint(119, 125, (nb, 1), generator=g, device=device, dtype=torch.int32)
    probs = torch.tensor([0.22, 0.2, 0.16, 0.13, 0.1, 0.09, 0.06, 0.04], device=device)
    mag = torch.multinomial(probs, nb * 32, replacement=True, generator=g).view(nb, 32)
    sign = torch.randint(0, 2, (nb, 32), generator=g, device=device) * 8
    nib = (mag + sign).to(torch.int32)
    codes = nib[:, :16] | (nib[:, 16:] << 4)
    return torch.cat([scale, codes], dim=1).to(torch.uint8).reshape(-1)
