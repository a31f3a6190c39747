"""SARA rollout collection on one GB300 (sm_103a): C-ABI library + thin Python binding.

The hot path (batched bf16 decode with tcgen05/TMEM GEMMs, GQA decode attention, fused
RMSNorm/RoPE epilogues, Gumbel-max sampling, and the on-device Algorithm 1 controller)
lives in libsara.so, built from csrc/ by build.py.  This package only marshals arguments.
"""
from .sara import (ABANDONED, COMMITTED, INCOMPLETE, SARA_EDEVICE, SARA_EINVAL, SARA_ENOMEM, SARA_ETIMEOUT, SARA_OK,
                   UNDRAWN, Handle, ModelCfg, SaraError, attention_decode, gemm_bf16, gemm_bf16_static, load,
                   model_cfg, sample, tau_fraction)

__all__ = ["Handle", "ModelCfg", "SaraError", "attention_decode", "gemm_bf16", "gemm_bf16_static", "load", "model_cfg", "sample",
           "tau_fraction", "UNDRAWN", "COMMITTED", "ABANDONED", "INCOMPLETE", "SARA_OK", "SARA_EINVAL", "SARA_ENOMEM",
           "SARA_ETIMEOUT", "SARA_EDEVICE"]
