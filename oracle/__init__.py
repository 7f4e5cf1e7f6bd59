"""CPU fp64 oracle of the AATC hot path -- test infrastructure only (see aatc_oracle)."""
