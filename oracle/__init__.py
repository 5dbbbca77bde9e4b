"""CPU oracle package (test infrastructure only; see decomoe_oracle)."""
