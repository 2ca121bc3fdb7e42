"""GB300-native hot path of structured suffix modeling (SSM) for block-wise
diffusion-LM decoding: selector, sparse step input, bidirectional attention
and confidence-based unmasking, as CUDA kernels for sm_103a behind the C ABI
of include/ssm.h.

``paper_2608_23167_gb300.ssm`` is the Python binding (ctypes over libssm.so);
``paper_2608_23167_gb300.workloads`` draws the seeded synthetic inputs.
The library is loaded on first use, not at import.
"""

__all__ = ["ssm", "workloads", "build_lib"]
