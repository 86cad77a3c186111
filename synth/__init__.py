"""Seeded synthetic inputs for the packed LM-head forward.

This package is the one piece shared by the CPU oracle's tests and the CUDA
path's tests and benchmark.  It only draws random numbers and lays them out
in the canonical packed layout; it performs none of the method's arithmetic
(no dequantisation, no products, no logits).
"""

from .inputs import (  # noqa: F401
    HeadShape,
    SHAPES,
    make_head,
    make_hidden,
    make_targets,
    head_nbytes_canonical,
    with_extreme_codes,
    make_dense_head,
    make_dense_head_device,
    make_test_matrix,
)
