"""Workload shapes: LoRA-adapted projections of 3B-class decoder layers.

The fine-tuning method adapts the q and v projections with r = 16, alpha = 16
(hyper-parameter table, "LoRA layers: q, v"); the workloads here adapt all
seven projections of a decoder layer (q, k, v, o, gate, up, down), which is a
superset of that setting.  Hidden sizes are those of Llama-3.2-3B
(3072 -> 3072 / 1024 / 8192) and Qwen-2.5-3B (2048 -> 2048 / 256 / 11008),
the two models of the paper's profiling setup.

Projections that read the same decoder activation share one input buffer:
q, k, v read the attention input; gate, up read the MLP input; o and down
read their own.  `group` names that buffer.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List


@dataclass(frozen=True)
class Proj:
    name: str
    d_in: int
    d_out: int
    group: int  # input-buffer id (projections with the same id share x)


@dataclass
class Workload:
    name: str
    cfg: int              # stream tag of the workload
    T: int                # tokens
    rank: int
    alpha: float
    projs: List[Proj] = field(default_factory=list)
    layers: int = 1
    zero_B: bool = False
    q4: bool = False      # base weights as 4-bit codes (Algorithm 1's on-the-fly dequantization)
    ckpt: bool = False    # checkpointed stack schedule (Algorithm 2): forward twice, backward once
    kind: str = "lora"    # "lora": adapted projections; "ce": LM-head cross entropy; "topk": similarity table
    vocab: int = 0        # ce: vocabulary size V
    hidden: int = 0       # ce: hidden size d
    topk: int = 0         # ce: k of the top-k table (0: full vocabulary)
    trainable: float = 1.0  # ce: fraction of trainable positions (prompt first, then response)
    cluster: int = 512    # ce: locality of the synthetic top-k table and targets

    @property
    def scale(self) -> float:
        return self.alpha / self.rank

    def flops(self) -> float:
        """Algorithmic FLOPs of one fwd+bwd over every projection and layer:
        4TKN (the two base contractions) + 6Tr(K+N) (the rank-r products);
        the frozen weight's gradient is never formed and not counted."""
        T, r = self.T, self.rank
        per = sum(4 * T * p.d_in * p.d_out + 6 * T * r * (p.d_in + p.d_out) for p in self.projs)
        return float(per * self.layers)


def llama_layer() -> List[Proj]:
    h, kv, f = 3072, 1024, 8192
    return [Proj("q", h, h, 0), Proj("k", h, kv, 0), Proj("v", h, kv, 0), Proj("o", h, h, 1),
            Proj("gate", h, f, 2), Proj("up", h, f, 2), Proj("down", f, h, 3)]


def qwen_layer() -> List[Proj]:
    h, kv, f = 2048, 256, 11008
    return [Proj("q", h, h, 0), Proj("k", h, kv, 0), Proj("v", h, kv, 0), Proj("o", h, h, 1),
            Proj("gate", h, f, 2), Proj("up", h, f, 2), Proj("down", f, h, 3)]


def single_small(zero_B: bool = False) -> Workload:
    """One 256 -> 256 projection, T = 128, r = 8, alpha = 16 (and its B = 0 twin)."""
    return Workload("single_T128_256x256_r8" + ("_B0" if zero_B else ""), 0, 128, 8, 16.0,
                    [Proj("lin", 256, 256, 0)], zero_B=zero_B)


def llama_q() -> Workload:
    """Llama-3.2-3B-shaped q projection, T = 512, r = 16, alpha = 32."""
    return Workload("llama3b_q_T512_r16", 1, 512, 16, 32.0, [Proj("q", 3072, 3072, 0)])


def llama_layer_T2048() -> Workload:
    """Seven projections of a Llama-3.2-3B-shaped layer, T = 2048, r = 16, alpha = 32."""
    return Workload("llama3b_layer_T2048_r16", 2, 2048, 16, 32.0, llama_layer())


def qwen_layer_T4096() -> Workload:
    """Seven projections of a Qwen-2.5-3B-shaped layer, T = 4096, r = 64, alpha = 128."""
    return Workload("qwen3b_layer_T4096_r64", 3, 4096, 64, 128.0, qwen_layer())


SWEEP_RANKS = (4, 8, 16, 32, 64, 128)
SWEEP_TOKENS = (256, 1024, 4096, 16384)


def llama_sweep(T: int, r: int) -> Workload:
    """Llama layer at (T, r) of the rank x token sweep; alpha = 2r keeps s = 2."""
    return Workload(f"llama3b_layer_T{T}_r{r}", 4, T, r, 2.0 * r, llama_layer())


def llama_stack28() -> Workload:
    """28 Llama layers' projections, T = 1024, r = 16, alpha = 32, forward of
    every layer first, then backward of every layer, from stored inputs."""
    return Workload("llama3b_stack28_T1024_r16", 5, 1024, 16, 32.0, llama_layer(), layers=28)


def llama_stack28_ckpt() -> Workload:
    """The 28-layer stack under the checkpointed schedule (Algorithm 2): every
    layer's forward saving nothing, then per layer from the last a re-forward
    and the backward."""
    return Workload("llama3b_stack28_T1024_r16_ckpt", 5, 1024, 16, 32.0, llama_layer(), layers=28, ckpt=True)


def llama_layer_T2048_q4() -> Workload:
    """The Llama layer at T = 2048, r = 16 with every base weight in 4-bit form."""
    return Workload("llama3b_layer_T2048_r16_q4", 6, 2048, 16, 32.0, llama_layer(), q4=True)


def llama_layer_T256(q4: bool = False) -> Workload:
    """The Llama layer at T = 256, r = 16: few tokens, so the weight bytes bound the contractions."""
    return Workload("llama3b_layer_T256_r16" + ("_q4" if q4 else ""), 7, 256, 16, 32.0, llama_layer(), q4=q4)


def llama_lm_head_ce() -> Workload:
    """Llama-3.2-3B LM head (V = 128256, d = 3072), T = 2048 positions of which
    the last 30 % are trainable, top-500 reduced vocabulary: the LM-head node of
    the paper's combined setting (top-k softmax approximation + logits masking)."""
    return Workload("llama3b_lmhead_ce_T2048_top500_mask30", 12, 2048, 1, 1.0, [], kind="ce", vocab=128256,
                    hidden=3072, topk=500, trainable=0.3)


def llama_lm_head_ce_full() -> Workload:
    """The same LM head with the full vocabulary (no top-k), logits masking only."""
    return Workload("llama3b_lmhead_ce_T2048_full_mask30", 12, 2048, 1, 1.0, [], kind="ce", vocab=128256,
                    hidden=3072, topk=0, trainable=0.3)


def llama_topk_table() -> Workload:
    """The top-k similarity table of a Llama-3.2-3B-sized embedding (V = 128256,
    d = 3072, k = 500, the paper's chosen k): a one-time precomputation."""
    return Workload("llama3b_topk_table_V128256_k500", 13, 0, 1, 1.0, [], kind="topk", vocab=128256, hidden=3072,
                    topk=500)


def topk_table_small() -> Workload:
    """A 40000-token table at d = 3072, k = 500: the sampled path on a few GB of device memory."""
    return Workload("topk_table_V40000_k500", 13, 0, 1, 1.0, [], kind="topk", vocab=40000, hidden=3072, topk=500)


BY_NAME = {
    "single": single_small,
    "single_B0": lambda: single_small(True),
    "llama_q": llama_q,
    "llama_layer": llama_layer_T2048,
    "qwen_layer": qwen_layer_T4096,
    "llama_stack28": llama_stack28,
    "llama_stack28_ckpt": llama_stack28_ckpt,
    "lm_head_ce": llama_lm_head_ce,
    "lm_head_ce_full": llama_lm_head_ce_full,
    "topk_table": llama_topk_table,
    "topk_table_small": topk_table_small,
    "llama_layer_q4": llama_layer_T2048_q4,
    "llama_layer_T256": llama_layer_T256,
    "llama_layer_T256_q4": lambda: llama_layer_T256(True),
}
