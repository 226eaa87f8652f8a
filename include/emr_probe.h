/*
 * emr_probe.h: ALU throughput probes of libemr (measurement support, not part
 * of the discovery path). The hot path is bound by the FP32 FMA pipe and the
 * special function unit (MUFU: exp2, reciprocal, sine) that its CPPN
 * activations use; these probes measure both rates on the running GPU so the
 * roofline can weight a MUFU operation by the measured FMA:MUFU ratio.
 */
#ifndef EMR_PROBE_H
#define EMR_PROBE_H

#include "emr.h"

#ifdef __cplusplus
extern "C" {
#endif

enum { EMR_PROBE_FFMA = 0, EMR_PROBE_EX2 = 1, EMR_PROBE_RCP = 2, EMR_PROBE_SIN = 3 };

/* Run `blocks` CTAs of 256 threads, each thread executing iters * 128
 * operations of kind op in 8 independent dependency chains, and time the
 * launch with CUDA events on `stream` (the call synchronises on that event).
 * *ops = operations executed, *ms = elapsed milliseconds. sink: device float
 * [blocks] that is written only to keep the chains live. Synchronous.
 * Errors: EMR_ERR_ARG, EMR_ERR_CUDA. */
emr_status emr_probe_alu(int32_t op, int32_t blocks, int32_t iters, double *ops, float *ms, float *sink,
                         void *stream);

#ifdef __cplusplus
}
#endif

#endif /* EMR_PROBE_H */
