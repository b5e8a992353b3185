"""Seeded synthetic inputs for the tests and the benchmark.

Input generators only -- no verification arithmetic lives here.  Both the
CPU oracle tests and the CUDA-path tests draw their inputs from this package.
"""
