"""CPU oracle for Heddle's batched candidate-plan pricing (test infrastructure only)."""
