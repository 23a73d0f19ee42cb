"""Efficient-Adam two-way quantized error-feedback round on GB300 (see include/ea.h)."""
