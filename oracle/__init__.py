"""Plain CPU oracle for the E2LLM deployment search (test infrastructure only)."""
