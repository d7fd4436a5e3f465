"""CPU oracle package (test infrastructure only; see snn_oracle)."""
