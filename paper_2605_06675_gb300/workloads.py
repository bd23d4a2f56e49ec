"""The synthetic KV-cache workloads this library is measured and tested on.

Shapes follow the models the paper evaluates (Sec. 4.1 "Models": GQA,
head_dim 128; Qwen3-8B 36 layers x 8 KV heads, Llama3.1-8B 32 x 8) plus a
70B-shaped long-context cache. Importance weights w are log-normal with the
sigma(ln w) the paper reports per model (App. R Table 19: Llama3.1-8B 0.74,
Qwen3-8B 0.76); bit sets follow the configurations named below.
"""
from __future__ import annotations

from dataclasses import dataclass

PER_TOKEN, PER_CHANNEL = 0, 1
PER_TOKEN_64, PER_TOKEN_128 = 2, 3     # TurboQuant's value / key groups (64 / 128 channels)


def mask_of(bits) -> int:
    m = 0
    for b in bits:
        m |= 1 << b
    return m


@dataclass(frozen=True)
class Workload:
    name: str
    L: int
    B: int
    H_kv: int
    H_q: int
    S: int
    dtype: str                 # "float16" | "bfloat16"
    k_grouping: int
    v_grouping: int
    hadamard: bool
    allowed: tuple
    avg_bits: float
    sigma_lnw: float
    value_dist: str            # "gaussian" | "student_t4"
    seed: int
    calib_T: int = 512
    k_quantizer: int = 0       # rq_quantizer: 0 min-max, 1 absmax (symmetric)
    v_quantizer: int = 0

    @property
    def g(self) -> int:
        return self.H_q // self.H_kv

    @property
    def n_components(self) -> int:
        return self.L * self.H_kv * 2

    @property
    def allowed_mask(self) -> int:
        return mask_of(self.allowed)

    def scaled(self, **kw) -> "Workload":
        d = dict(self.__dict__)
        d.update(kw)
        return Workload(**d)


TINY = Workload("tiny_1L_S1024_fp16", L=1, B=1, H_kv=8, H_q=32, S=1024, dtype="float16",
                k_grouping=PER_CHANNEL, v_grouping=PER_TOKEN, hadamard=False,
                allowed=(2, 3, 4), avg_bits=3.0, sigma_lnw=0.5, value_dist="gaussian", seed=0)

LLAMA3_8B_32K = Workload("llama3_8b_L32_B8_S32768_kivi", L=32, B=8, H_kv=8, H_q=32, S=32768,
                         dtype="bfloat16", k_grouping=PER_CHANNEL, v_grouping=PER_TOKEN,
                         hadamard=False, allowed=(2, 3, 4), avg_bits=2.5, sigma_lnw=0.74,
                         value_dist="gaussian", seed=1)

QWEN3_8B_8K = Workload("qwen3_8b_L36_B16_S8192_hadamard", L=36, B=16, H_kv=8, H_q=32, S=8192,
                       dtype="bfloat16", k_grouping=PER_TOKEN, v_grouping=PER_TOKEN,
                       hadamard=True, allowed=(2, 3, 4, 5, 6, 7, 8), avg_bits=4.0,
                       sigma_lnw=0.76, value_dist="gaussian", seed=2)

CALIB_SWEEP = Workload("calib_sweep_L32_H8_T512", L=32, B=1, H_kv=8, H_q=32, S=512,
                       dtype="bfloat16", k_grouping=PER_CHANNEL, v_grouping=PER_TOKEN,
                       hadamard=False, allowed=(2, 3, 4), avg_bits=2.5, sigma_lnw=0.74,
                       value_dist="gaussian", seed=3)

LONG_70B_128K = Workload("llama70b_L80_B1_S131072_kivi", L=80, B=1, H_kv=8, H_q=64, S=131072,
                         dtype="bfloat16", k_grouping=PER_CHANNEL, v_grouping=PER_TOKEN,
                         hadamard=False, allowed=(2, 3, 4, 8), avg_bits=3.0, sigma_lnw=0.5,
                         value_dist="student_t4", seed=4)

ALL = [TINY, LLAMA3_8B_32K, QWEN3_8B_8K, CALIB_SWEEP, LONG_70B_128K]
