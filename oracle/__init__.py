"""fp64 CPU oracle of the evicted-KV decode step -- test infrastructure only."""
