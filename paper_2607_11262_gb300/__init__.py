"""Batched graph-driven tile-graph simulation (GPU-Tile-Sim backend) for GB300.

* ``workloads`` -- seeded synthetic tile graphs and design-point tables;
* ``gts``       -- binding of libgts (include/gts.h), the CUDA implementation;
* ``build``     -- nvcc build of libgts for sm_103a.
"""
