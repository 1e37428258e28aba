"""CPU oracle for the Forward-Forward train step and predict (test infrastructure only)."""
