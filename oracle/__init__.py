"""CPU oracle of the FedOptima server-side hot path (test infrastructure only)."""
