"""CPU oracle (test infrastructure only; see evo_oracle)."""
