"""CPU oracle of the DeepShift operators: test infrastructure only (see deepshift_oracle)."""
