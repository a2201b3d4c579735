"""Float64 CPU oracle of the SPADE verify step (test infrastructure only)."""
