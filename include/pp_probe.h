/*
 * pp_probe.h -- benchmark helper library libpp_probe.so (not part of the
 * planner's ABI in prefixplace.h, and with no counterpart in the paper).
 */
#ifndef PP_PROBE_H
#define PP_PROBE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/*
 * pp_probe_read -- reads the device buffer `buf` (`bytes` bytes, 16-byte
 * aligned, a multiple of 16) `iters` times with 16-byte loads that bypass L1,
 * on all SMs of the current device.  A buffer that fits in L2 gives the L2
 * read bandwidth that the roofline of the DP's skip-row gathers is quoted
 * against; a buffer far larger than L2 gives the HBM read bandwidth.  `sink`
 * (device, 8 bytes) only keeps the loads live.  Asynchronous on `stream`
 * (a cudaStream_t, NULL = the legacy default stream).
 * Returns 0, 1 for a bad argument (null pointer, misaligned buffer or size,
 * iters < 0), 2 when a CUDA call fails.
 */
int pp_probe_read(const void *buf, size_t bytes, int32_t iters, uint64_t *sink, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* PP_PROBE_H */
