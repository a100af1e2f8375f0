"""SOAP optimizer step (arXiv 2607.20548, Alg. 1) batched over a model's weights on one GB300.

The compute path is libsoap.so (hand-written CUDA for sm_103a behind the C ABI of
include/soap.h, and the paper's Muon step behind include/muon.h); ``soap`` is its ctypes
binding and ``workloads`` draws the synthetic inputs.
"""
from .soap import (MuonOptimizer, SoapError, SoapOptimizer, Shape, default_hparams, load_library, soap_create,
                   soap_gemm, soap_qr, soap_state_get, soap_state_set, soap_step)

__all__ = ["MuonOptimizer", "SoapError", "SoapOptimizer", "Shape", "default_hparams", "load_library",
           "soap_create", "soap_gemm", "soap_qr", "soap_state_get", "soap_state_set", "soap_step"]
