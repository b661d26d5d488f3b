"""GB300-native BOM (Backpropagated Output Momentum) task-space momentum pass."""
