/*
 * sim_peaks.h - measured on-chip ceilings for the roofline of the batched scheduler simulator
 * (libsim.so).  The paper has no counterpart: this is a measurement utility.
 */
#ifndef SIM_PEAKS_H_
#define SIM_PEAKS_H_

#ifdef __cplusplus
extern "C" {
#endif

/*
 * sim_measure_peaks: measure, on the current device, the two ceilings of the simulation kernel's
 * roofline, each by a full-occupancy microbenchmark timed with CUDA events (best of three after a
 * warm-up, about 0.1 s in all):
 *   out[0]  integer operations per second: independent chains of one 32-bit add and one 32-bit
 *           xor per link, which issue as two integer ALU instructions;
 *   out[1]  shared-memory read bytes per second: conflict-free 16-byte loads per lane (512 bytes,
 *           four wavefronts, per warp instruction);
 *   out[2], out[3]  the two kernels' times in milliseconds.
 * `out` is HOST memory of 4 doubles.  Allocates a few KB of device memory for the duration of
 * the call.  Returns 0, -1 (out is NULL), -4 (a CUDA call failed) or -6 (allocation failed).
 */
int sim_measure_peaks(double *out);

#ifdef __cplusplus
}
#endif

#endif /* SIM_PEAKS_H_ */
