"""fp64 CPU oracle of the TreeFlash drafting path (test infrastructure only)."""
