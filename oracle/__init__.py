"""fp64 CPU oracle for the ECOKV eviction pass (test infrastructure only)."""
