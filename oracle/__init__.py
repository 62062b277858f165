"""Reference CPU simulator and brute-force checker (test infrastructure only)."""
