"""CPU oracle for the SAKI hot path (test infrastructure only; see saki_oracle)."""
