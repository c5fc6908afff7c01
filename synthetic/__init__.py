"""Seeded synthetic inputs (no attention arithmetic) shared by the oracle and the CUDA path."""
