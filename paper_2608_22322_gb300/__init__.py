"""AL-quantized optimizer steps for GB300 (sm_103a).

Adaptive Log-Space (AL8/AL16) coded non-negative states and uniform 8-bit
(UF8) signed momentum, decoded, updated and re-encoded in fused CUDA kernels
for AdamW, Adafactor, CAME and APOLLO. The kernels live in the C-ABI library
libalq.so (include/alq.h); `binding` exposes each entry point under the same
name for torch CUDA tensors; `optim` wraps the steps as torch.optim
optimizers (AdamW, Adafactor, CAME, Apollo). The binding is loaded on first
use, so the synthetic-workload module can be imported without the library.
"""
from . import workloads  # noqa: F401

_BINDING_NAMES = {
    "al_encode", "al_decode", "uf8_encode", "uf8_decode", "al_adamw_step",
    "AdamWPlan", "al_adafactor_step", "al_came_step", "al_apollo_step",
    "al_num_blocks", "al_state_bytes", "al_workspace_size", "version", "AlqError",
    "AL_OP_ADAFACTOR", "AL_OP_CAME", "AL_OP_APOLLO", "ApolloPlan", "FactoredPlan",
}


def __getattr__(name):
    if name in _BINDING_NAMES:
        from . import binding
        return getattr(binding, name)
    raise AttributeError(name)
