"""fp64 CPU oracle of the GMC compression step: test infrastructure only (see gmc_oracle)."""
