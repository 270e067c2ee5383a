"""The fp64 CPU oracle of the PIPO pair step (test infrastructure only)."""
