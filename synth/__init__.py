"""Seeded synthetic inputs shared by the tests, bench.py and the oracle's callers.

This package holds shapes and random draws only: no step of the method
(masking, ELBO, bound, gradient, advantage normalisation) is computed here.
"""
from .workloads import (CONFIGS, SWEEP_NT, Workload, make_inputs, make_old_head,  # noqa: F401
                        make_per_sample_hidden, zipf_targets)
