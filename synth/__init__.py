"""Seeded synthetic inputs for the LoCA hot path (see ``synth.inputs``)."""

from .inputs import WORKLOADS, Workload, host_inputs, host_probe_pairs, device_inputs, scaled

__all__ = ["WORKLOADS", "Workload", "host_inputs", "host_probe_pairs", "device_inputs", "scaled"]
