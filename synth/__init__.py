"""Seeded synthetic workloads shared by the CUDA harness and the CPU oracle."""
