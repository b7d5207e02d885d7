/*
 * maps_bench.h -- test and benchmarking aids of libmaps.so.  Not part of the
 * scheduler's interface (include/maps.h): a scheduler never needs them, and
 * with their defaults they change nothing.  The paper has no counterpart.
 */
#ifndef MAPS_BENCH_H
#define MAPS_BENCH_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* `before` and `after` are CUDA events (cudaEvent_t, created by the caller,
 * passed as void *).  Every later SNAPSHOT maps_dispatch call made by this
 * thread records them on its stream right before and right after its scoring
 * kernel (after the candidates have been bucketed by horizon tile), so a
 * caller can time the scoring kernel alone.  An event between two launches
 * costs the programmatic overlap there.  NULL, NULL turns it off.  Results
 * are unaffected.  Returns MAPS_OK (0). */
int maps_set_dispatch_events(void *before, void *after);

/* Exercises the bounded waits of maps_order_local's global form (the form
 * taken when arrival is not non-decreasing along the index and the call is
 * larger than one block): on the current device, later calls let tile `tile`
 * of every radix pass publish nothing to the decoupled look-back, and every
 * look-back wait gives up after `spin_limit` polls (0: the library default).
 * The tile after the withheld one then waits until the limit, records
 * MAPS_E_TIMEOUT (read with maps_check) and carries on; the order of that
 * call is wrong, every write stays inside the outputs, and the device stays
 * usable.  tile = -1, spin_limit = 0 restores the normal behaviour.  Calls in
 * flight must have finished before the settings change.  Returns MAPS_OK or
 * MAPS_E_CUDA. */
int maps_test_withhold_lookback(int32_t tile, uint32_t spin_limit);

/* Exercises the bounded grid barriers of maps_order_local's finishing kernel
 * (the cooperative kernel that ranks or merges the long queues, or runs the
 * global form's passes): on the current device, later calls make block
 * `block` of that kernel return at once, so the other blocks' first barrier
 * waits until the limit maps_test_withhold_lookback sets (0 there: the
 * library default), records MAPS_E_TIMEOUT and ends each block without
 * another write.  The order of that call is wrong; what it wrote before the
 * barrier stays inside its outputs and workspace.  block = -1 restores the
 * normal behaviour.  Calls in flight must have finished before the setting
 * changes.  Returns MAPS_OK or MAPS_E_CUDA. */
int maps_test_absent_block(int32_t block);

/* Exercises the bounded grid barrier of maps_calibrate's cooperative kernel
 * (calibration sets above 8,192 residuals): on the current device, later
 * calls make block `block` of that kernel return at once, so the other
 * blocks' barrier gives up after `spin_limit` polls (0: the library default),
 * records MAPS_E_TIMEOUT (read with maps_check) and ends each block without
 * another write: q and the bounds of that call are not written.  block = -1,
 * spin_limit = 0 restores the normal behaviour.  Calls in flight must have
 * finished before the settings change.  Returns MAPS_OK or MAPS_E_CUDA. */
int maps_test_calibrate_absent_block(int32_t block, uint32_t spin_limit);

#ifdef __cplusplus
}
#endif
#endif /* MAPS_BENCH_H */
