"""Plain CPU oracle for the RelaySum step (test infrastructure only)."""
