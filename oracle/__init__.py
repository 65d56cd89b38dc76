"""fp64 CPU oracle of PACE's hot path: test infrastructure only (see pace_oracle)."""
