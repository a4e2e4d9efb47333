"""fp64 CPU oracle of the DBW iteration: test infrastructure only (see dbw_oracle)."""
