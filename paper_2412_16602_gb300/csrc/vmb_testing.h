// vmb_testing.h - test-only controls of libvmb, not part of the public ABI
// (include/vmb.h does not declare them and production callers never call
// them).  The tests use them to run every tile shape and chunk length of the
// scans, which the planners would otherwise pick by problem size alone.
//
// The overrides are process-wide and take effect on the next plan; calls made
// while an override is set (by any thread) get the forced plan.  Restore the
// defaults (-1 / 0) when done.
#pragma once

#include <stddef.h>

#include "vmb.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Force the full scan's tile shape (0..15 for 16 states; taken modulo the
 * number of shapes of the padded state count) and, for the look-back shapes,
 * the number of L-chunks (<= 1: one chunk).  shape < 0 restores the planner.
 * Ignored under VMB_FLAG_B_ZOH, which has one shape.  Returns 0. */
int vmb_testing_force_full_plan(int shape, int chunks);

/* Force the chunk length of the channel-mean scan (32, 64 or 128; 0 restores
 * the planner).  Returns 0, or 1 for another value (nothing changes). */
int vmb_testing_force_mean_chunk(int tc);

/* Workspace bytes of the plan one scan call with these exact flags would run
 * (vmb_scan_workspace_bytes returns the larger over the two Bbar forms).
 * 0 for invalid arguments. */
size_t vmb_testing_plan_workspace_bytes(int path, unsigned flags, int B, int K, int D, int N, int H, int W,
                                        vmb_dtype dtype);

#ifdef __cplusplus
}
#endif
