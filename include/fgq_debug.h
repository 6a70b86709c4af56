/*
 * fgq_debug.h -- test and benchmark controls of libfgq (not needed to use the library).
 *
 * Each control is per host thread: it affects only the calls that thread makes, so a
 * test or benchmark that sets one cannot change the kernels another thread's calls run.
 * Paper counterpart: none.
 */
#ifndef FGQ_DEBUG_H_
#define FGQ_DEBUG_H_

#include <stdint.h>

#include "fgq.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Contraction kernel families (see fgq_set_path / fgq_last_path). */
typedef enum {
  FGQ_PATH_AUTO = 0,   /* choose per shape: the few-row path for small GEMMs; with
                          fixed-point alphas the dense tensor-core path where it applies;
                          else the tensor cores where the shape is covered (G = 4 only with
                          at least 64 filters per conv group), else the CUDA cores */
  FGQ_PATH_SIMT = 1,   /* CUDA-core path: dp4a group sums, one FMA per group */
  FGQ_PATH_TC = 2,     /* tensor-core path (tcgen05): G in {64, 128} with K-tiles aligned to
                          the group; G = 4 with a block-diagonal activation operand
                          (Cg a multiple of 64) */
  FGQ_PATH_GEMV = 3,   /* few-row path for GEMMs with P <= 8 (8-bit activations, Kred a
                          multiple of 16, G >= 4): one warp per filter row streams the
                          weights once; the automatic choice for such calls */
  FGQ_PATH_DENSE = 4   /* dense tensor-core path (tcgen05, any G, 8-bit activations, Cg a
                          multiple of 64): the alphas are folded into fp16 weights
                          alpha(m, k / G) * t[m][k] built per call, and one dense
                          contraction replaces the per-group multiplies.  Fixed-point alphas
                          fold into integer weights |a t| <= 255: the automatic choice for
                          fgq_gemm_qa / fgq_conv2d_qa (bounds in fgq.h).  With fp32 alphas
                          forcing this path returns FGQ_ERR_UNSUPPORTED unless
                          fgq_debug_allow_split_fold(1) was called on the thread: the alphas
                          are then split per filter row into two fp16 parts after scaling the
                          row's largest alpha into [2^14, 2^15), about 22 bits of alpha, and
                          the fp32 accumulator rounds once per 16 reduction elements -- a
                          numerical ablation of folding, outside the fgq_gemm tolerance. */
} fgq_path;

/*
 * Restricts this thread's contraction calls to one kernel family (FGQ_PATH_AUTO restores
 * the default per-shape choice).  A forced path that cannot run a shape makes the call
 * return FGQ_ERR_UNSUPPORTED.  Returns the previous setting, or -1 for an unknown path.
 */
int fgq_set_path(int path);

/* The kernel family (fgq_path) the most recent contraction call on this host thread used. */
int fgq_last_path(void);

/*
 * Shortens every mbarrier wait of the tensor-core contraction kernels launched by this
 * thread to about `us` microseconds (us < 0 restores the kernels' own limit of about one
 * second per wait), so that a test can make a wait run out on purpose: the kernel then
 * records FGQ_ERR_TIMEOUT, each role leaves its loop, and the kernel waits -- with its
 * normal limits, which this setting never shortens -- for the copies and MMAs it issued,
 * frees its tensor memory and returns.  Returns the previous setting.
 */
int64_t fgq_debug_set_wait_limit_us(int64_t us);

/*
 * Lets FGQ_PATH_DENSE run calls with fp32 alphas on this thread through the split-fp16
 * ablation (allow != 0), outside the fgq_gemm tolerance; 0 restores FGQ_ERR_UNSUPPORTED.
 * Returns the previous setting.
 */
int fgq_debug_allow_split_fold(int allow);

/*
 * Runs the G = 4 tensor-core output kernel of this thread's calls on CTA pairs (on != 0: two
 * SMs share each 64-filter x 256-position tile through cta_group::2 MMAs) or on single CTAs
 * (0, the default: 32-filter tiles), the same results either way.  Returns the previous
 * setting.
 */
int fgq_debug_cta_pairs(int on);

/*
 * At most k (1 .. 8, clamped) group ranges per output tile in this thread's G >= 64
 * tensor-core calls; returns the previous limit (default 8).  A layer with fewer output tiles
 * than SMs splits each tile's groups into ranges and adds the ranges' partial sums into the
 * output: the same sum in another fp32 rounding order, and with more than two ranges not
 * bit-reproducible from run to run.  k = 1 keeps whole tiles (one rounding order, the one
 * the fused requantizing entries use).
 */
int fgq_debug_max_ksplit(int k);

/* Group ranges per tile of this thread's last G >= 64 tensor-core call (1: whole tiles). */
int fgq_debug_last_ksplit(void);

/*
 * The CUDA runtime error (a cudaError_t value) behind the last FGQ_ERR_CUDA that a kernel
 * launch of this thread returned, 0 if none; reading it clears it.  `name` receives the
 * runtime's name of that error (at most `len` bytes including the terminator) when non-null.
 */
int fgq_debug_last_cuda_error(char* name, size_t len);

#ifdef __cplusplus
}
#endif

#endif /* FGQ_DEBUG_H_ */
