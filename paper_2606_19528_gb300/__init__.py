"""GB300 (sm_103a) LoRA-adapted linear layer: forward and backward with the
base weight frozen, as a C-ABI CUDA library (include/lora.h) with a thin
ctypes binding (`lora`).  `synth` draws the seeded bf16 inputs and
`workloads` names the layer shapes; neither holds any LoRA arithmetic.
"""
__all__ = ["lora", "synth", "workloads", "build"]
