"""Archer (arXiv 2608.08086) per-step hot path for one GB300 (sm_103a).

Submodules:
  archer      ctypes binding of libarcher's C ABI (include/archer.h); importing it
              loads the CUDA library and fails loudly when it is missing
  trajectory  the state-anchored decoding loop (Algorithm 1) over the C ABI,
              host-driven or one step graph per step (refresh branch on the
              device), with checkpoint / restore
  synth       seeded synthetic inputs (no arithmetic of the method)
  build       nvcc build of libarcher.so for sm_103a
The C-ABI functions are re-exported lazily: ``from paper_2608_08086_gb300
import archer_attn_step`` loads libarcher.so on first use.
"""
_ABI = ("archer_attn_step", "archer_prompt_refresh", "archer_attn_workspace_size", "archer_decode_scores",
        "archer_decode_scores_workspace_size", "archer_should_refresh", "archer_cache_rewrite",
        "archer_decoder_update", "archer_scatter_rows", "archer_check_device", "archer_version", "make_shape",
        "attn_workspace", "scores_workspace", "StepGraph", "ArcherError")


def __getattr__(name):
    if name in _ABI:
        from . import archer
        return getattr(archer, name)
    raise AttributeError(name)
