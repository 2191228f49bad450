"""GB300-native DARD step: state-masked attention and confidence scoring (arXiv 2608.26574).

The compute path is the C-ABI library ``libdard.so`` (CUDA kernels for sm_103a) built from
``csrc/``; ``binding`` marshals torch tensors into its calls. ``workloads`` holds the
seeded synthetic input generators.
"""
