"""GB300-native WbG128 (b = 3, 4) weight-only quantized linear layer (LAQuant, arXiv 2605.08755).

The product is ``liblaq.so`` (C ABI in include/laq.h, CUDA for sm_103a).  This package is its
thin Python binding (``_lib``) plus the decode-step weight pass harness (``weight_pass``) that
captures the 252 per-token GEMV launches of a Qwen3-shaped decoder into one CUDA graph.
"""
from ._lib import (EXPORTS, Chain, GemmConfig, LaqError, chain_status, chain_workspace,  # noqa
                   laq_chain_workspace_bytes, laq_gemm_chain, laq_gemm_plan, laq_gemm_wxg128,
                   laq_pack, laq_quantize_rtn, laq_unpack, lib, packed_bytes)

__all__ = ["EXPORTS", "Chain", "GemmConfig", "LaqError", "chain_status", "chain_workspace",
           "laq_chain_workspace_bytes", "laq_gemm_chain", "laq_gemm_plan", "laq_gemm_wxg128",
           "laq_pack", "laq_quantize_rtn", "laq_unpack", "lib", "packed_bytes"]
