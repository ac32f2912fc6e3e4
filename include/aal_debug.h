/*
 * aal_debug.h -- test hooks of libaal.so.
 *
 * Not part of the computation: one lets a test make one of the library's bounded device
 * waits run out on purpose, so that the timeout path can be checked on a GPU without a
 * fault, a trap or a hang; the other exposes a host-side launch decision so that it can be
 * checked without a GPU.
 */
#ifndef AAL_DEBUG_H_
#define AAL_DEBUG_H_

#include <stdint.h>

#include "aal.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Arms the next forward pass that streams logits through a TMA ring (aal_loss_fwd or
 * aal_seq_loss_fwd on rows a multiple of 16 bytes, including the token-id form, or the
 * reference-draft pass of aal_grpo_from_loss) to leave the completion barrier of its
 * `chunk`-th ring copy (counted from 0 in each CTA's stream) unarmed: the consumers of that
 * chunk wait on a phase that nothing completes.  Every wait of that kernel, and of later ones, gives up
 * after `wait_limit_ns` (0 restores the default of 1 s); the kernel then records
 * AAL_ERR_TIMEOUT in the workspace status word, walks its remaining loops without waiting,
 * drains its copies and returns, so aal_check_device_status() reports AAL_ERR_TIMEOUT and
 * the context stays usable.  The results of that call are not valid.  A negative
 * `chunk` arms nothing.  The chunk setting is consumed by the next forward or GRPO call. */
AAL_API void aal_debug_fail_next_forward(int64_t chunk, uint64_t wait_limit_ns);

/* Windows per solo CTA in the launch of aal_loss_fwd_bwd's fused kernels, as the host chooses
 * it: N windows of K rows, G groups of K CTAs (each group finishes one window per row time)
 * and S spare CTAs (each takes whole windows, K row times each).  Returns an m >= 0 with
 * m S <= N that minimises the launch's length in row times, max(ceil((N - m S) / G), m K),
 * and 0 whenever no solo CTAs (m = 0) is as short; 0 when G <= 0 or S <= 0.  Pure host
 * arithmetic: no GPU is touched. */
AAL_API int64_t aal_debug_solo_windows(int64_t N, int32_t K, int32_t G, int32_t S);

/* The shortest row (in bytes, V times the element size) for which aal_loss_fwd_bwd and
 * aal_seq_loss_fwd_bwd launch their fused kernels; shorter rows run the two calls inside them,
 * which are faster there (the fused form pays a window exchange per row, and a short row has
 * little streaming to hide it behind).  The same threshold picks the streamed forward's geometry
 * for bf16 rows (shorter rows: 8 consumer warps and two CTAs an SM; also in the streamed sampling
 * reward), so the forward inside the fused call and the separate forward agree.  A negative value
 * restores the default (AAL_FUSED_MIN_ROW_BYTES_DEFAULT); 0 fuses every row the fused kernels
 * take, so that a test can exercise them on short rows.  Either way the results of the one-call
 * entry points are those of their two calls, bit for bit. */
#define AAL_FUSED_MIN_ROW_BYTES_DEFAULT 131072
AAL_API void aal_debug_fused_min_row_bytes(int64_t bytes);

#ifdef __cplusplus
}
#endif

#endif /* AAL_DEBUG_H_ */
