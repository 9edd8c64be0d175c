"""Seeded synthetic workloads for one global round of distributed sign momentum.

This module is pure data: the parameter layouts (tensor lists) and the
hyper-parameters of the five measured workloads.  It holds none of the
method's arithmetic, so both the CPU oracle and the CUDA path may read it.

Parameter layouts follow the GPT-2 family of Table 1 (Sec. 5, model
configurations): Small 768/12, Medium 1024/24, Large 1280/36, plus XL
1600/48; vocabulary 50257 and context 1024 (Sec. 5, experiments set-up).
The language-model head is tied to the token embedding, so it is not a
separate tensor.  Only the element count, the kind and the synthetic
gradient scale of each tensor matter on this path.

Synthetic gradients stand in for the OpenWebText backward pass, which is
not available: g_i[e] = s_T*(u(seed, step, e) - 1/2) + (0.1 s_T)*(u(seed, i, e) - 1/2)
with u a 24-bit counter-based hash.  The generator itself is implemented
separately by each side (see the oracle and the CUDA grad-fill kernel).
"""
from __future__ import annotations

import dataclasses
from typing import List, Tuple

# Tensor kinds (same numbering as the C-ABI's DSM_KIND_*).
KIND_WEIGHT = 0
KIND_BIAS = 1
KIND_LN_W = 2
KIND_LN_B = 3

# Base optimizers and sign modes (same numbering as the C-ABI).
BASE_ADAMW = 0
BASE_SGDM = 1
SIGN = 0          # deterministic sign, Eq. (model-update)
RSIGN_ZERO = 1    # randomized sign, Eq. (rand-sign-2): 0 or sign(v)
RSIGN_PM = 2      # randomized sign, Eq. (rand-sign-1): -sign(v) or sign(v)
F32 = 0
BF16 = 1
# Global steps: Algorithm 1 and the variants of the ablations (Sec. 5)
GLOBAL_SIGN_MOMENTUM = 0
GLOBAL_SLOWMO = 1
GLOBAL_SIGNED_SLOWMO = 2
GLOBAL_LOOKAHEAD = 3
GLOBAL_ADAMW = 4
# Flags: FUSED_ROUND is an execution option (the results do not depend on it);
# RESET_LOCAL_STATE selects a variant of the method (every round starts each
# worker's base-optimizer state from zero and restarts AdamW's step count).
FLAG_FUSED_ROUND = 1
FLAG_RESET_LOCAL_STATE = 2

VOCAB = 50257
CONTEXT = 1024


@dataclasses.dataclass(frozen=True)
class Tensor:
    name: str
    numel: int
    kind: int
    grad_scale: float
    wd: int = 1


@dataclasses.dataclass(frozen=True)
class HParams:
    base: int = BASE_ADAMW
    lr: float = 6e-4          # gamma: local learning rate, also gamma_t of the global step
    b1: float = 0.9           # local AdamW beta1
    b2: float = 0.95          # local AdamW beta2
    eps: float = 1e-8
    wd: float = 0.1           # local decoupled weight decay (AdamW only)
    mu: float = 0.9           # SGD-momentum coefficient (0 => plain SGD)
    g_b1: float = 0.9         # global beta1, Eq. (ut-update)
    g_b2: float = 0.99        # global beta2, Eq. (mom-update)
    g_eta: float = 1e-3       # global learning rate eta, Eq. (model-update)
    g_wd: float = 0.1         # global decoupled weight decay lambda
    sign_mode: int = SIGN
    rsign_B: float = 1e-2     # bound B of Eqs. (rand-sign-1/2)
    grad_dtype: int = F32
    seed: int = 0
    global_mode: int = 0      # GLOBAL_* below
    g_eps: float = 1e-8       # epsilon of the global AdamW step
    flags: int = 0            # FLAG_* above


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    tensors: Tuple[Tensor, ...]
    n: int
    tau: int
    rounds: int
    hp: HParams

    @property
    def d(self) -> int:
        return sum(t.numel for t in self.tensors)


def gpt2_layout(layers: int, d_model: int, mlp: int, w_scale: float = 1e-3,
                small_scale: float = 1e-4) -> Tuple[Tensor, ...]:
    """GPT-2 parameter list in nanoGPT order (Conv1D-transposed weights)."""
    D, M = d_model, mlp
    t: List[Tensor] = [
        Tensor("wte", VOCAB * D, KIND_WEIGHT, w_scale),
        Tensor("wpe", CONTEXT * D, KIND_WEIGHT, w_scale),
    ]
    for l in range(layers):
        p = f"h{l}."
        t += [
            Tensor(p + "ln_1.weight", D, KIND_LN_W, small_scale),
            Tensor(p + "ln_1.bias", D, KIND_LN_B, small_scale),
            Tensor(p + "attn.c_attn.weight", D * 3 * D, KIND_WEIGHT, w_scale),
            Tensor(p + "attn.c_attn.bias", 3 * D, KIND_BIAS, small_scale),
            Tensor(p + "attn.c_proj.weight", D * D, KIND_WEIGHT, w_scale),
            Tensor(p + "attn.c_proj.bias", D, KIND_BIAS, small_scale),
            Tensor(p + "ln_2.weight", D, KIND_LN_W, small_scale),
            Tensor(p + "ln_2.bias", D, KIND_LN_B, small_scale),
            Tensor(p + "mlp.c_fc.weight", D * M, KIND_WEIGHT, w_scale),
            Tensor(p + "mlp.c_fc.bias", M, KIND_BIAS, small_scale),
            Tensor(p + "mlp.c_proj.weight", M * D, KIND_WEIGHT, w_scale),
            Tensor(p + "mlp.c_proj.bias", D, KIND_BIAS, small_scale),
        ]
    t += [Tensor("ln_f.weight", D, KIND_LN_W, small_scale),
          Tensor("ln_f.bias", D, KIND_LN_B, small_scale)]
    return tuple(t)


def flat_layout(d: int, scale: float) -> Tuple[Tensor, ...]:
    return (Tensor("flat", d, KIND_WEIGHT, scale),)


ADAMW_HP = HParams()
SGDM_HP = HParams(base=BASE_SGDM, lr=1e-2, mu=0.9, wd=0.0,
                  sign_mode=RSIGN_ZERO, rsign_B=1e-2)

# The five measured workloads.  Hyper-parameters that a workload leaves
# unstated inherit the flat workload's values (local AdamW lr 6e-4,
# betas (0.9, 0.95), eps 1e-8, wd 0.1; global betas (0.9, 0.99), eta 1e-3,
# lambda 0.1).
WORKLOADS = {
    "flat1m": Workload("flat1m: flat fp32 d=1048576, n=4, tau=4, AdamW, sign",
                       flat_layout(1 << 20, 1e-2), n=4, tau=4, rounds=3, hp=ADAMW_HP),
    "gpt2s": Workload("gpt2s: GPT-2 small 124M, n=4, tau=12, AdamW fp32 grads, sign",
                      gpt2_layout(12, 768, 3072), n=4, tau=12, rounds=5, hp=ADAMW_HP),
    "gpt2m": Workload("gpt2m: GPT-2 medium 355M, n=8, tau=24, AdamW bf16 grads, sign",
                      gpt2_layout(24, 1024, 4096), n=8, tau=24, rounds=5,
                      hp=dataclasses.replace(ADAMW_HP, grad_dtype=BF16)),
    "gpt2l": Workload("gpt2l: GPT-2 large 774M, n=8, tau=12, SGD-momentum fp32 grads, "
                      "randomized sign B=1e-2",
                      gpt2_layout(36, 1280, 5120), n=8, tau=12, rounds=3, hp=SGDM_HP),
    "gpt2xl": Workload("gpt2xl: GPT-2 XL 1.56B, n=4, tau=24, AdamW bf16 grads, sign",
                       gpt2_layout(48, 1600, 6400), n=4, tau=24, rounds=3,
                       hp=dataclasses.replace(ADAMW_HP, grad_dtype=BF16)),
}

# The workload the throughput line is quoted on: the largest one GPU holds (about 100 GB of state).
BENCH_WORKLOAD = "gpt2xl"

