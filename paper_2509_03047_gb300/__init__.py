"""libflashrec for GB300 (sm_103a): the restoration sweep of FlashRecovery
(arXiv 2509.03047, Sec. III-E) -- per-chunk fingerprint, pack, unpack+verify
and diff over a rank's model and optimizer state, in hand-written CUDA.

``paper_2509_03047_gb300.flashrec`` is the ctypes binding of the C ABI in
``include/flashrec.h``; importing it fails loudly if the library is not built.
``shards`` restores ZeRO / FSDP shards from differently sharded replicas,
``steptag`` holds the step-tag recovery controller (Sec. III-E), ``overhead``
the recovery-overhead model (Eq. 1-5), and ``synth`` generates the seeded
synthetic workloads.
"""
