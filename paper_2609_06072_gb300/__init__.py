"""GB300 (sm_103a) grouped adapter execution for ACE (arxiv 2609.06072).

The compute path is the C-ABI CUDA library ``libace.so`` (include/ace.h);
``paper_2609_06072_gb300.ace`` is its ctypes binding and
``paper_2609_06072_gb300.workloads`` draws the seeded synthetic inputs.
"""
__all__ = ["ace", "workloads"]
