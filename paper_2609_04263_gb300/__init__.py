"""GB300-native packed low-bit KV-cache attention step with fused LoRA Q/K/V.

The compute path is the C-ABI library libkvq.so (hand-written sm_103a CUDA);
`kvq` is its thin ctypes binding.  Importing this package does not load the
library; the first call into `kvq` does, and fails loudly if it is missing.
"""
