"""GB300-native SJD-PAC verify-and-draft hot path (speculative Jacobi decoding
with proactive drafting and adaptive continuation).

The compute path is the CUDA library libsjd.so (C ABI, include/sjd.h);
`paper_2603_18599_gb300.sjd` is its thin Python binding.
"""
