/* gem_sim.h -- the asynchronous-system simulator around the GEM commit path.
 *
 * The paper's workers commit asynchronously; which worker commits at each tick of the
 * global clock, and with what staleness, follows from an implicit queueing model
 * (Introduction, Eq. staleness: s_t = theta_{t - tau_t}, expected staleness n - 1 under
 * a homogeneous model).  On one GPU that behaviour is simulated: a seeded schedule fixes
 * the commit order, and a segment planner groups consecutive commits by distinct workers,
 * whose gradients can then be computed together because none of their snapshots changes
 * inside the group.
 *
 * Random numbers: SplitMix64 (Steele, Lea & Flood, OOPSLA 2014).  The stream for
 * (seed, id) starts at mix64(seed * 0x9E3779B97F4A7C15 + id) and its c-th output is
 * mix64(start + 0x9E3779B97F4A7C15 (c + 1)).  Host-only functions; they return 0, or -1
 * on an invalid argument.
 */
#ifndef GEM_SIM_H
#define GEM_SIM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Uniform tick (stream id 10): at tick t the worker floor(n u / 2^32) commits, u the top
 * 32 bits of output t.  order [T] receives the workers; tau [T] (may be NULL) the
 * staleness of each commit, t minus the tick of the worker's previous commit minus one
 * (t for its first commit: it pulled theta_0).  Requires n >= 1, T >= 0. */
int gem_schedule_uniform(uint64_t seed, int n, int T, int32_t* order, int32_t* tau);

/* Exponential-service queue (stream id 10 + 1): worker w's j-th gradient takes
 * -ln(1 - u) / rate time units, u = (output (w << 32) | j) >> 11 times 2^-53; the worker
 * that finishes first commits next (ties to the lower id) and starts its next gradient.
 * Same outputs as gem_schedule_uniform.  Requires rate > 0. */
int gem_schedule_queue(uint64_t seed, int n, int T, double rate, int32_t* order,
                       int32_t* tau);

/* Segment planner: cuts order [T] into maximal runs of consecutive commits by distinct
 * workers.  seg_start [T + 1] receives the first commit of each segment followed by T;
 * returns the number of segments S (seg_start[0..S]), or -1 on an invalid argument. */
int gem_plan_segments(const int32_t* order, int T, int n, int32_t* seg_start);

#ifdef __cplusplus
}
#endif

#endif /* GEM_SIM_H */
