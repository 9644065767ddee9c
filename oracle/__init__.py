"""CPU oracle of the routed block (test infrastructure only; see cer_oracle)."""
