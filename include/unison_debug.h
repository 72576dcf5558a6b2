/* unison_debug.h -- test hooks of the ranking call (not in the library).
 *
 * These entry points exist only in the separate test library built by
 * paper_2609_09643_gb300.native.build_debug() (libunison_rank_debug.so:
 * the ranking call compiled with UNISON_DEBUG_HOOKS).  The default library,
 * libunison.so, neither exports them nor contains the hooks.  The paper has
 * no counterpart: they let a test show that a bounded device wait of the
 * ranking kernel runs out, reports itself, and leaves the GPU usable.
 *
 * In the test library every bounded wait of the ranking kernel gives up
 * after a few thousand polls instead of more than a second.
 */
#ifndef UNISON_DEBUG_H
#define UNISON_DEBUG_H

#ifdef __cplusplus
extern "C" {
#endif

/* For the following unison_rank_batch calls: the kernel's wait for the
 * thresholds of set flag_set first waits on a flag that nothing sets, and
 * its first wait for a tile of set mbar_set first waits on an mbarrier that
 * nothing arrives at.  Both bounded waits run out; the set's counts[3] then
 * reads UNISON_ERR_TIMEOUT, and the kernel goes on to its ordinary waits, so
 * its other outputs are still the exact ranking.  -1 turns a hook off.
 * Returns UNISON_OK, or UNISON_ERR_CUDA if the hooks could not be set. */
int unison_debug_rank_wait_hooks(int flag_set, int mbar_set);

#ifdef __cplusplus
}
#endif

#endif /* UNISON_DEBUG_H */
