"""CPU fp64 oracle of the parareal network (test infrastructure only)."""
