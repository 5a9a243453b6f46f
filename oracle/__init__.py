"""CPU oracle for the revisit path (test infrastructure only; see prcr_oracle)."""
