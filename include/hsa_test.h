/*
 * hsa_test.h -- test hooks of libhsa (not needed by applications).
 *
 * The attention kernel bounds every pipeline wait (about one second) and, when
 * one runs out, records HSA_ERR_TIMEOUT, stops issuing work, drains its own
 * copies and tensor-core operations, frees its tensor memory and returns, so
 * the CUDA context stays usable.  This hook lets a test drive that path on a
 * GPU without any fault: it withholds one internal signal so that a wait can
 * never complete.  The paper has no counterpart.
 */
#ifndef HSA_TEST_H
#define HSA_TEST_H

#ifdef __cplusplus
extern "C" {
#endif

/* mode 0: normal operation (default).
 * mode 1: in every bf16 hsa_active_attention launch that follows, each CTA
 *         never loads its first value tile, so the bounded wait for it runs
 *         out; the call then reports HSA_ERR_TIMEOUT through
 *         hsa_get_device_error and its output is unspecified.
 * Process-wide, host side only; returns the previous mode, or
 * HSA_ERR_INVALID_ARG (-1) for an unknown mode. */
int hsa_test_inject_attention_stall(int mode);

#ifdef __cplusplus
}
#endif

#endif /* HSA_TEST_H */
