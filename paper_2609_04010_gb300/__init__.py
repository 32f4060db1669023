"""GB300-native verify step of lossless diffusion-drafted decoding (Psi-Spec).

The compute path is the CUDA library ``libspecverify.so`` (sm_103a) behind the C ABI
declared in ``include/spec_verify.h``; :mod:`paper_2609_04010_gb300.binding` marshals
torch tensors into it.  :mod:`paper_2609_04010_gb300.workloads` draws seeded synthetic
inputs.  Importing the package loads nothing; the binding loads the library on first use
and raises if it is missing.
"""
