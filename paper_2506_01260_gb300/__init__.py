"""GB300-native (sm_103a) stage-boundary codec of Subspace Networks (arXiv 2506.01260).

The CUDA library (``libsn.so``, C ABI in ``include/sn.h``) compresses
residual-stream activations and activation gradients onto an orthonormal basis
U at a pipeline boundary, reconstructs them on the other side, and projects the
residual-writing weights onto span(U).  ``paper_2506_01260_gb300.sn`` is the
thin Python binding; ``workloads`` synthesises seeded inputs.
"""
__all__ = ["sn", "workloads"]
