"""GB300 (sm_103a) implementation of MeBP's LoRA training step (arxiv 2510.03425).

The compute lives in ``libmebp.so`` (CUDA kernels behind the C ABI of include/mebp.h);
``paper_2510_03425_gb300.mebp`` is the ctypes binding and ``paper_2510_03425_gb300.model``
holds the torch-side weight/buffer plumbing around it.
"""
