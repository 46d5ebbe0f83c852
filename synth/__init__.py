"""Seeded synthetic telemetry inputs (no accounting arithmetic)."""
