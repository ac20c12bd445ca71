"""CPU oracle for the W4A16 linear layer (test infrastructure only)."""
