"""GB300-native group-sparse linear layer y = x (W (.) M)^T (GroupMask, Sec. 2.1, Eq. 1).

Submodules:
  groupsparse  ctypes binding of libgroupsparse.so (pack / linear / unpack); loads the CUDA library
  workload     seeded synthetic inputs (weights, group masks, activations)
  build        nvcc build of libgroupsparse.so for sm_103a

Importing the package itself loads nothing; `import paper_2609_33977_gb300.groupsparse`
loads the compiled library and fails loudly if it is missing.
"""
