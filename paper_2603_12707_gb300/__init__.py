"""GB300-native paged KV cache and batched single-token decode attention for
multimodal LLM serving (the language-decoding hot path of HeteroServe,
arXiv 2603.12707).

The compute path is libkvdecode.so (hand-written CUDA for sm_103a, C ABI in
include/kvdecode.h); ``kvdecode`` is its ctypes binding, ``workloads`` draws
seeded synthetic inputs and ``harness`` drives a decode session through the
C ABI.  Importing this package loads nothing; the library is loaded on first
use and its absence is an error.
"""
__all__ = ["kvdecode", "workloads", "harness"]
