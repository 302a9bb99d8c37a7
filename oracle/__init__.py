"""CPU oracle of the WAMachine hot path (test infrastructure; see wam_oracle)."""
