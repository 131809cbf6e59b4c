"""GB300 (sm_103a) implementation of the training-side token pass of
calibrated importance sampling (CIS), arxiv 2609.32444.

``binding``  thin Python binding of libcis (include/cis.h)
``synth``    seeded synthetic workloads
``build``    nvcc build of libcis.so
"""
