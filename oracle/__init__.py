"""fp64 CPU oracle of the BeaconKV compression step (test infrastructure only)."""
