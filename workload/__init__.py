"""Seeded synthetic workloads shared by the oracle tests, the GPU tests and the bench."""
from .gen import (CONFIGS, make_config, make_problem, query_slice, query_subset,
                  simulate_online, arrivals, feature_layout, to_bf16_bits,
                  bf16_bits_to_f32, XF_ID, XF_LOG1P, XF_LOG)
