"""CPU oracle of the ALR slot-loss path (test infrastructure; never used by the product)."""
