/*
 * whtmix.h -- C ABI of the WHTMix token mixer for NVIDIA GB300 (sm_103a).
 *
 * The operation (paper Section III-B, Eq. 1-4, "Walsh-Hadamard Token Mixer"): for each plane
 * X_b [N, C] of a batch (tokens x channels) and one gain matrix G [N, C],
 *
 *     Y_b = H_N ( G (.) (H_N X_b H_C) ) H_C / (N C)
 *
 * where H_n is the n x n Sylvester-Hadamard matrix, (H_n)_{ij} = (-1)^{popcount(i & j)}.  With the
 * orthonormal transform W = H_N (.) H_C / sqrt(N C) this is Y = W (G (.) W X): a forward 2D
 * Walsh-Hadamard transform, a per-frequency gain, and the inverse transform (W is its own
 * inverse).  The paper's learnable log-domain gains g_c, g_t are the rank-1 case
 * G = exp(g_t) exp(g_c)^T; the input/output projections W_in, W_out (Eq. 1, Eq. 4) are dense
 * GEMMs outside this call.  The paper zero-pads the token axis to a power of two before the
 * transform; here N and C must already be powers of two (pad on the caller's side).
 *
 * The backward (not printed in the paper, which trains the block end to end; it follows from
 * the map being linear in X and in G and from W being symmetric):
 *
 *     dX_b = H_N ( G (.) (H_N dY_b H_C) ) H_C / (N C)
 *     dG   = sum_{b = 0 .. B-1, ascending} (H_N X_b H_C) (.) (H_N dY_b H_C) / (N C)
 *
 * Conventions for every call below
 *   Layout      X, Y, dY, dX: row-major contiguous [B, N, C] (c fastest, then n, then b).
 *               G, dG: row-major contiguous [N, C].  All are DEVICE pointers unless stated.
 *   dtype       WHTMIX_F32:  X/Y/dY/dX float32, G/dG float32, orthonormal (1/(N C)), fp32 math.
 *               WHTMIX_BF16: X/Y/dY/dX bfloat16, G/dG float32, orthonormal, fp32 math, the
 *                            outputs rounded to nearest-even once at the store.
 *               WHTMIX_I32:  X/Y/dY/dX int32, G/dG int32, UNnormalised (no 1/(N C)), every
 *                            operation wraps modulo 2^32 -- the result is exact and independent
 *                            of the order of the butterfly stages.
 *   Shapes      B >= 0, N >= 1 and C >= 1 powers of two, N*C <= 2^30 elements per plane,
 *               B*N*C <= 2^60.  B = 0: the forward returns WHTMIX_OK without touching anything
 *               (null data pointers are accepted); the backward sets dG to zero (the sum over no
 *               planes) and touches nothing else, so only dgains must be valid.
 *   Alignment   every pointer must be 16-byte aligned.
 *   Aliasing    y == x (and dx == dy) is allowed and computes in place.  Any other overlap
 *               between an output and an input or another output returns WHTMIX_ERR_ALIAS.
 *   Streams     `stream` is a cudaStream_t (NULL = the legacy default stream).  Calls are
 *               asynchronous on that stream; all argument checks run on the host before anything
 *               is enqueued, and a call that returns an error has enqueued nothing and written
 *               nothing.  Faults of the device code surface at the caller's next synchronisation.
 *   Ownership   the caller owns every pointer it passes.  The plain calls keep a workspace per
 *               (device, stream), allocated stream-ordered on first use and grown on demand;
 *               whtmix_release_workspaces() frees them.  The cache is keyed by the stream's
 *               handle, so call it before destroying a stream that plain calls used (a stream
 *               created later may receive the same handle).  The _ex calls use the caller's
 *               workspace instead and allocate nothing.
 *   Threads     calls on different streams may run concurrently from different host threads.
 *               Two calls that share a workspace (same stream, or the same _ex buffer) must be
 *               ordered by that stream.
 */
#ifndef WHTMIX_H
#define WHTMIX_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define WHTMIX_API __attribute__((visibility("default")))
#else
#define WHTMIX_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum { WHTMIX_F32 = 0, WHTMIX_BF16 = 1, WHTMIX_I32 = 2 } whtmix_dtype_t;

typedef enum {
    WHTMIX_OK = 0,
    WHTMIX_ERR_INVALID_ARG = 1, /* null pointer where data is needed, B < 0, N < 1 or C < 1   */
    WHTMIX_ERR_BAD_SHAPE = 2,   /* N or C not a power of two, N*C > 2^30, B*N*C too large     */
    WHTMIX_ERR_BAD_DTYPE = 3,   /* dtype not one of whtmix_dtype_t                             */
    WHTMIX_ERR_MISALIGNED = 4,  /* a pointer is not 16-byte aligned                            */
    WHTMIX_ERR_ALIAS = 5,       /* partial overlap between an output and another buffer        */
    WHTMIX_ERR_CUDA = 6,        /* a CUDA runtime call failed: see whtmix_last_cuda_error()    */
    WHTMIX_ERR_TIMEOUT = 7,     /* a bounded device-side wait expired (reported by whtmix_sync) */
    WHTMIX_ERR_NO_DEVICE = 8,   /* no CUDA device, or the current device is not sm_103         */
    WHTMIX_ERR_WORKSPACE = 9    /* _ex call: workspace null, misaligned or smaller than needed */
} whtmix_status_t;

/* Forward mixer.  Section III-B, Eq. 1-4 (the map between W_in and W_out).
 *   x      [B, N, C] input planes (dtype)            gains  [N, C] G (float32, int32 for I32)
 *   y      [B, N, C] output planes (dtype); may equal x.
 * Returns a whtmix_status_t.  One kernel launch on `stream` (two for some shapes, five per plane
 * group for planes of more than 2^26 elements; none when B = 0). */
WHTMIX_API int whtmix_forward(const void *x, const void *gains, void *y, int64_t B, int64_t N, int64_t C,
                   int dtype, void *stream);

/* Forward mixer with a 16-bit exchange: the map of whtmix_forward (Section III-B, Eq. 1-4), same
 * arguments, where only the storage between the three-phase kernel's phases differs.  Planes of
 * 2^14 .. 2^23 elements that run the three-phase kernel (fp32 or bf16 I/O) keep their butterflies
 * and the gain in fp32 but round the intermediate plane to bf16 (nearest, ties to even) at the
 * two points where it crosses between SMs: after the row bits and after the column bits.  That
 * halves the workspace traffic through L2.  Each rounding moves a value by at most 2^-8 of itself,
 * so the output's relative L2 error grows by at most 2^-8 (max|G| / min|G| + 1) over
 * whtmix_forward's (measured: 2.3e-3 with fp32 I/O, 2.9e-3 with bf16 I/O, gains near 1); it is
 * not bit-identical to whtmix_forward.  Every other shape (int32, planes held on chip, planes
 * below 2^14 or above 2^23 elements) runs exactly what whtmix_forward runs.  The paper has no
 * such variant (it trains under bf16 autocast and states no kernel). */
WHTMIX_API int whtmix_forward_x16(const void *x, const void *gains, void *y, int64_t B, int64_t N, int64_t C,
                       int dtype, void *stream);

/* Backward mixer: both gradients of the forward map.
 *   x      [B, N, C] the forward input              gains [N, C] G
 *   dy     [B, N, C] upstream gradient dL/dY          dx   [B, N, C] dL/dX (may equal dy)
 *   dgains [N, C] dL/dG, float32 (int32 for I32), OVERWRITTEN (not accumulated into); the sum
 *          over b runs in ascending b, so the result is bit-reproducible run to run.
 * dgains may not overlap x, dy, dx or gains. */
WHTMIX_API int whtmix_backward(const void *x, const void *gains, const void *dy, void *dx, void *dgains,
                    int64_t B, int64_t N, int64_t C, int dtype, void *stream);

/* Workspace size in bytes for the _ex calls (backward != 0 for whtmix_backward_ex).  Writes
 * *out_bytes; the size depends only on the arguments. */
WHTMIX_API int whtmix_workspace_bytes(int64_t B, int64_t N, int64_t C, int dtype, int backward, size_t *out_bytes);

/* Same as whtmix_forward / whtmix_backward with a caller-owned device workspace of at least
 * whtmix_workspace_bytes() bytes, 256-byte aligned.  Its first 256 bytes hold a device-wide
 * barrier (32-bit words 0, 1, 3, 4: arrival counters; word 2: error; word 5: barrier sequence
 * number) and must be zero before the first call that uses the buffer (cudaMemset), and again
 * after a call whose wait gave up (non-zero error word); a call that completes leaves the header
 * in the state the next call continues from.  Calls sharing a workspace must be ordered on one
 * stream. */
WHTMIX_API int whtmix_forward_ex(const void *x, const void *gains, void *y, int64_t B, int64_t N, int64_t C,
                      int dtype, void *workspace, size_t workspace_bytes, void *stream);
WHTMIX_API int whtmix_backward_ex(const void *x, const void *gains, const void *dy, void *dx, void *dgains,
                       int64_t B, int64_t N, int64_t C, int dtype, void *workspace,
                       size_t workspace_bytes, void *stream);

/* Forward that allocates no device memory, for callers that may not allocate while they run:
 * a process whose device memory is owned up front by an outside allocator or framework, a
 * real-time loop where an allocation could stall or fail at the wrong moment, a plugin handed
 * only its input and output buffers.  The paper has no counterpart.  Same arguments as
 * whtmix_forward, and the same kernels for the shape (plane groups limited to the scratch below),
 * so the results are those of whtmix_forward bit for bit.
 * Scratch: the kernels keep their barrier header and intermediate planes in a fixed device array
 * of 16 MiB + 256 B defined by the library; every GPU that loads the library holds it until the
 * process exits.  Limit: planes of N*C <= 2^13 elements need no scratch; larger planes need
 * N*C <= 2^22 (4 Mi fp32 elements), else the call returns WHTMIX_ERR_WORKSPACE and enqueues
 * nothing.  B = 0 is a no-op.  The first call on each device looks up the array's device address
 * with a CUDA runtime call; make that first call before any stream capture.  A call enqueues two
 * 4-byte memsets (the barrier's arrival counts) and one kernel.  All calls share the array, which
 * keeps the previous call's contents: calls whose kernels can overlap on the GPU (different
 * streams, or different host threads) race on it -- order them on one stream.  A bounded
 * device-wide wait that gives up sets the array's error word, which stays set (later calls keep
 * it) until whtmix_sync reports it as WHTMIX_ERR_TIMEOUT and clears it. */
WHTMIX_API int whtmix_forward_noalloc(const void *x, const void *gains, void *y, int64_t B, int64_t N,
                                      int64_t C, int dtype, void *stream);

/* Token-axis zero padding inside the library (Section III-B: a non-power-of-two token count is
 * zero-padded to a power of two before H_N, and the padded outputs are discarded).  x, y, dy and
 * dx hold only the first N_valid tokens of each plane, [B, N_valid, C] row-major; the mixer acts on
 * the plane padded with zero rows to [N, C] (N a power of two, 0 <= N_valid <= N) and gains /
 * dgains are [N, C].  Same results as padding by hand, calling whtmix_forward / whtmix_backward
 * and cropping the output rows (the upstream gradient of the discarded rows is zero).  The fast
 * kernels read only the stored rows and write only the kept rows when every stored plane starts
 * 16-byte aligned (N_valid * C * sizeof(dtype) a multiple of 16); other shapes pad and crop through
 * copies in the library workspace.  N_valid = N is exactly whtmix_forward / whtmix_backward;
 * N_valid = 0 or B = 0 stores nothing (the backward sets dgains to zero).  Other rules as for
 * whtmix_forward / whtmix_backward. */
WHTMIX_API int whtmix_forward_padded(const void *x, const void *gains, void *y, int64_t B, int64_t N_valid, int64_t N,
                                     int64_t C, int dtype, void *stream);
WHTMIX_API int whtmix_backward_padded(const void *x, const void *gains, const void *dy, void *dx, void *dgains,
                                      int64_t B, int64_t N_valid, int64_t N, int64_t C, int dtype, void *stream);

/* The paper's own gain parameterisation (Section III-B, Eq. 2-3): per-frequency log gains for the
 * token axis, g_t [N], and the channel axis, g_c [C], fp32, applied in the WHT domain as
 * G[n, c] = exp(g_t[n]) * exp(g_c[c]).  Because the channel and token mixes act on different axes,
 * the sequential Eq. 2 -> Eq. 3 form equals the 2D map with this rank-one G, and these calls
 * compute exactly what whtmix_forward_padded / whtmix_backward_padded compute with
 * G = fp32(expf(g_t[n]) * expf(g_c[c])), token padding included (N_valid as there; N_valid = N for
 * none).  dtype is WHTMIX_F32 or WHTMIX_BF16 (WHTMIX_I32 returns WHTMIX_ERR_BAD_DTYPE).  x, y, dy,
 * dx: 16-byte aligned; g_t, g_c, dg_t, dg_c: 4-byte aligned; device memory owned by the caller.
 * Forward: for the planes the fast kernel covers (2^14 <= N*C <= 2^23) with 2 <= C <= 2^13 (2^14
 * for N*C = 2^23), the gains are computed inside the kernel from two small tables of exp values
 * and G never exists in memory; other shapes build G in the library workspace first.
 * Backward: dx as whtmix_backward_padded with that G; dg_t[n] = sum_c dG[n, c] G[n, c] and
 * dg_c[c] = sum_n dG[n, c] G[n, c] with dG = sum_b (W X_b) o (W dY_b) (the chain rule through
 * the exponentials), each a fixed-order sum accumulated in float64 (bit-reproducible).  dg_t and
 * dg_c are overwritten.  B = 0 or N_valid = 0: the forward is a no-op; the backward sets dg_t and
 * dg_c to zero.  Aliasing as for whtmix_forward / whtmix_backward (y == x and dx == dy allowed). */
WHTMIX_API int whtmix_forward_separable(const void *x, const float *g_t, const float *g_c, void *y, int64_t B,
                                        int64_t N_valid, int64_t N, int64_t C, int dtype, void *stream);
WHTMIX_API int whtmix_backward_separable(const void *x, const float *g_t, const float *g_c, const void *dy, void *dx,
                                         float *dg_t, float *dg_c, int64_t B, int64_t N_valid, int64_t N, int64_t C,
                                         int dtype, void *stream);

/* Token-wise channel projection on the tensor cores: z[t, :] = x[t, :] w^T for T tokens of C
 * channels, x [T, C] bf16, w [C, C] bf16 stored (out, in) like a linear layer's weight, z [T, C]
 * in out_dtype (WHTMIX_BF16, rounded to nearest even, or WHTMIX_F32); fp32 accumulation.  These
 * are the block's W_in and W_out (Section III-B, Eq. 1 and Eq. 4).  C must be 64, 128 or 256
 * and T*C <= 2^60 (WHTMIX_ERR_BAD_SHAPE otherwise).  z may be x itself for bf16 output; no other
 * overlap.  16-byte aligned device pointers; T = 0 is a no-op. */
WHTMIX_API int whtmix_project(const void *x, const void *w, void *z, int64_t T, int64_t C, int out_dtype,
                              void *stream);

/* The whole mixer block of Section III-B, Eq. 1-4, forward: Z = X W_in^T, M = the mixer of Z with
 * gains G (as whtmix_forward), Y = M W_out^T, per token row; x, y [B, N, C] bf16, w_in, w_out
 * [C, C] bf16 (out, in), gains [N, C] fp32; arithmetic is fp32 and M is rounded to bf16 before
 * W_out (the block's activation).  dtype must be WHTMIX_BF16; C 64, 128 or 256.  y may be x itself.
 * C = 128 with 2^21 <= N*C <= 2^23: one launch on `stream` (the projections fused into the mixer's
 * row phases; Z stays fp32).  Other shapes: three launches (projection, mixer, projection), each in
 * place in y, Z also rounded to bf16. */
WHTMIX_API int whtmix_block_forward(const void *x, const void *w_in, const void *gains, const void *w_out, void *y,
                                    int64_t B, int64_t N, int64_t C, int dtype, void *stream);

/* Backward of the whole mixer block (whtmix_block_forward's map, Section III-B, Eq. 1-4) for the
 * upstream gradient dY of its output: with Z = X W_in^T and M = mix(Z) recomputed in bf16 (the
 * forward's activations),
 *     dM = dY W_out,   (dZ, dG) = whtmix_backward at (Z, G, dM),   dX = dZ W_in,
 *     dW_out = sum over every token t of dY[t]^T M[t],   dW_in = sum over t of dZ[t]^T X[t].
 *   x, dy, dx [B, N, C] bf16 (dx may be dy itself); w_in, w_out [C, C] bf16 (out, in); gains [N, C]
 *   fp32; dw_in, dw_out [C, C] fp32 and dgains [N, C] fp32, all three OVERWRITTEN.
 * dM and dZ are rounded to bf16 (activation gradients); the weight gradients run on the tensor
 * cores in fp32 and are summed over token chunks in a fixed order, so every output is the same bit
 * for bit run to run.  dtype must be WHTMIX_BF16; C 64, 128 or 256.  B = 0 sets the three gain and
 * weight gradients to zero.  About fifteen launches on `stream`; the intermediates live in a second
 * library-managed workspace of the stream. */
WHTMIX_API int whtmix_block_backward(const void *x, const void *w_in, const void *gains, const void *w_out,
                                     const void *dy, void *dx, void *dw_in, void *dgains, void *dw_out, int64_t B,
                                     int64_t N, int64_t C, int dtype, void *stream);

/* Synchronises `stream` and reports device-side failures of the calls enqueued on it since the
 * previous whtmix_sync: WHTMIX_ERR_TIMEOUT if a bounded device-wide wait gave up (the library
 * then resets that workspace's barrier), WHTMIX_ERR_CUDA if the synchronisation itself failed,
 * WHTMIX_OK otherwise.  Checked: the library-managed workspace of `stream` and, on the current
 * device, the fixed scratch of whtmix_forward_noalloc (pass the stream those calls used, so that
 * they have finished).  Caller-owned _ex workspaces are the caller's to read (error word at byte
 * offset 8). */
WHTMIX_API int whtmix_sync(void *stream);

/* Frees every library-managed workspace on the current device (synchronises the device). */
WHTMIX_API int whtmix_release_workspaces(void);

/* Static description of a status code; never NULL. */
WHTMIX_API const char *whtmix_status_string(int status);

/* The cudaError_t of the last CUDA failure seen by this host thread (0 if none). */
WHTMIX_API int whtmix_last_cuda_error(void);

/* Which kernel plan a shape uses: 1 = one tile per plane group (N*C <= 2^13), 2 = three
 * passes through the workspace in one launch (2^13 < N*C <= 2^26), 3 = five passes, one launch
 * each (seven for the backward), through the workspace (2^26 < N*C <= 2^30); 0 for an invalid
 * shape.  (The fp32 / bf16 forward of a 2^14- or 2^15-element plane with full gains, and of a
 * 2^16-element plane in batches of 80 or more, runs one plane per CTA instead, in the SM's tensor
 * memory, without the workspace.) */
WHTMIX_API int whtmix_plan(int64_t N, int64_t C);

#ifdef __cplusplus
}
#endif

#endif /* WHTMIX_H */
