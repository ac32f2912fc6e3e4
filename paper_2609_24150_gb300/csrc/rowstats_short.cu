// Forward row statistics for short rows (bf16 rows under the fused call's threshold, 128 KB by
// default): the kernels of rowstats_stream.cu with 8 consumer warps and a 4 x 24 KB ring, two
// CTAs an SM.  A row of V = 32000 is three chunks of the default ring, so its fixed costs (the
// CTA reductions, the hand-over to the finisher warp, the ring's refill at each row start) weigh
// on the row; two CTAs an SM hide one CTA's row end behind the other's streaming, and the rows in
// flight (2 x 152 x 2 x 64 KB) stay far inside L2.  Measured at V = 32000 (N = 2048, K = 5):
// the two-pass forward 0.375 -> 0.325 ms, the one-pass forward 0.236 -> 0.207 ms; at V = 128256
// the default geometry is the faster one (5.85 against 6.07 ms), so long rows keep it.
//
// The warps fold different elements than the default geometry's, so the statistics differ from
// it in the last bits; the caller uses one geometry per row length for every call (the loss
// forward, the fused call's threshold, the streamed sampling reward), so the calls that must
// agree bit for bit still do.
#define AAL_STREAM_WARPS 8
#define AAL_STREAM_SLOT_KB 24
#define AAL_STREAM_CTAS 2
#define AAL_ROWSTATS_STREAM_NAME launch_rowstats_stream_short
#define AAL_REWARD_STREAM_NAME launch_reward_stream_short
#include "rowstats_stream.cu"
