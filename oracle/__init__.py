"""CPU oracle for the group-sparse linear layer (test infrastructure only; see groupsparse_oracle)."""
