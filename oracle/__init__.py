"""CPU oracle for the interaction-network edge classifier (test infrastructure only)."""
