"""fp64 CPU oracle of the LoRA-adapted linear layer.

Test infrastructure only: the tests, the smoke check and the benchmark's CPU
baseline arm are its only users; the CUDA library never imports it.
"""
from .lora_oracle import (lora_forward, lora_backward, lora_forward_rows,  # noqa: F401
                          lora_backward_dx_rows, lora_adapter_grads, lora_step,
                          unpack_q4, dequant_q4)
from .lm_head_oracle import reduced_vocab, ce_forward_backward  # noqa: F401,E402
from .topk_oracle import normalize_rows, similarities, topk_table  # noqa: F401,E402
