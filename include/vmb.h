/*
 * vmb.h - C ABI of the GB300 (sm_103a) library for the VMamba SS2D selective
 * scan and its channel-mean variant VMeanba (arXiv 2412.16602).
 *
 * The SS2D module (App. A, "VMamba" paragraph) is cross-scan -> selective scan
 * per direction -> cross-merge.  The selective scan is the discretised,
 * input-dependent state space model of App. A, Eqs. 3, 4 and 6.  VMeanba
 * (Sec. 2.2, Eq. 9) replaces the scan's inputs (Abar, Bbar u, C) by their mean
 * over the inner channel axis, runs one recurrence, and broadcasts the result
 * back to every channel.
 *
 * Conventions shared by every call
 *   - All tensor pointers are caller-owned DEVICE memory, dense row-major.
 *     The library allocates nothing, and scratch memory (the look-back
 *     workspace of the scans) is passed in by the caller.  The one exception
 *     is vmb_selective_scan_fwd_noalloc, for callers that cannot allocate:
 *     its scratch is a fixed array built into the library (one per device),
 *     and it keeps a host-side table of that array's device addresses.
 *   - Every call only validates its arguments and enqueues kernels on
 *     `stream`; it never synchronises (except vmb_read_status) and never
 *     throws or aborts.  Validation errors return before any launch, with no
 *     side effects.  A failed launch returns VMB_ERR_CUDA.
 *   - Shapes: B batch, K scan directions, D inner channels (d_inner), N state
 *     size (d_state), H x W the feature map, L = H*W the sequence length.
 *     A zero B, K, D, H or W is an empty problem: the call returns VMB_OK and
 *     launches nothing.  Negative sizes, or sizes whose element counts do
 *     not fit in int64, return VMB_ERR_INVALID_ARG.
 *   - dtype is the storage type of x/xs/u/delta/Bs/Cs/y/out (fp32 or bf16);
 *     A, Dskip and delta_bias are always fp32; arithmetic and the scan state
 *     are always fp32.  bf16 outputs are rounded to nearest even.
 *   - Pointers must be aligned to their element size (VMB_ERR_MISALIGNED
 *     otherwise).  16-byte aligned rows take the vectorised load path; other
 *     layouts take an element-wise path that gives the same results.
 *   - Outputs must not alias inputs.
 *   - Calls are thread-safe.  Scan calls that share one workspace must not
 *     overlap in time (order them on one stream).
 *   - Kernels are launched with programmatic stream serialization
 *     (programmatic dependent launch): their blocks may be scheduled while
 *     the previous kernel of the stream is finishing, and each waits
 *     (griddepcontrol.wait) for that kernel to complete before it reads or
 *     writes global memory.  (The exception: a warp-specialised full scan
 *     whose grid is smaller than one wave is launched normally, so that its
 *     blocks spread over every SM.)  Stream order is therefore kept for any
 *     preceding work; a caller's own kernel launched after a vmb call with
 *     the same attribute must likewise wait before touching vmb outputs.
 */
#ifndef VMB_H
#define VMB_H

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    VMB_OK = 0,
    VMB_ERR_INVALID_ARG = 1, /* null pointer, bad size or flag */
    VMB_ERR_MISALIGNED = 2,  /* pointer not aligned to its element size (workspace: 256 B) */
    VMB_ERR_UNSUPPORTED = 3, /* valid request this build does not implement (e.g. N > 16) */
    VMB_ERR_WORKSPACE = 4,   /* workspace missing or smaller than vmb_scan_workspace_bytes() */
    VMB_ERR_CUDA = 5,        /* a CUDA runtime call or kernel launch failed */
    VMB_ERR_TIMEOUT = 6,     /* device side: a look-back wait gave up (read via vmb_read_status) */
    VMB_ERR_BOUNDS = 7       /* device side: an index check failed (bounds-checked builds only) */
} vmb_status;

typedef enum { VMB_F32 = 0, VMB_BF16 = 1 } vmb_dtype;

/* Scan flags (bitwise OR). */
#define VMB_FLAG_SOFTPLUS 0x1u  /* delta = softplus(delta_raw + delta_bias) (Eq. 6); else raw + bias */
#define VMB_FLAG_B_ZOH 0x2u     /* Bbar = (exp(delta A) - 1) / A * B, zero-order hold (Eq. 4);
                                   else the Euler form Bbar = delta * B */
#define VMB_FLAG_SKIP_MEAN 0x4u /* vmb_mean_scan_fwd only: skip term = mean_d(Dskip_c u_d),
                                   broadcast; else per channel Dskip_c * u_d */
/* Test hook, never set in production: the first L-chunk of every sequence of
 * a multi-chunk scan does not publish its state, so that the look-back waits
 * of its successors run out (bounded, about 0.2 s) and the call reports
 * VMB_ERR_TIMEOUT through vmb_read_status; in the warp-specialised full scan
 * the first stage of every tile is never handed to the compute warps, so
 * their waits and then the copy warp's run out (bounded, about 1 s each) and
 * the call reports VMB_ERR_TIMEOUT.  No effect on other single-chunk plans. */
#define VMB_FLAG_TEST_SUPPRESS_PUBLISH 0x40000000u

/* Scan path selector for vmb_scan_workspace_bytes. */
#define VMB_PATH_FULL 0
#define VMB_PATH_MEAN 1

/*
 * vmb_cross_scan - SS2D cross-scan (App. A, "VMamba": unfold the H x W map
 * along four directions into four 1-D sequences).
 *   x   [B, D, H, W]       input map
 *   xs  [B, 4, D, L]       output sequences: direction 0 reads the map row by
 *                          row, 1 column by column, 2 and 3 are 0 and 1 reversed:
 *     xs[b,0,d,l] = x[b,d,l/W,l%W]      xs[b,1,d,l] = x[b,d,l%H,l/H]
 *     xs[b,2,d,l] = xs[b,0,d,L-1-l]     xs[b,3,d,l] = xs[b,1,d,L-1-l]
 * A pure permutation: results are bit-exact copies of x.
 */
vmb_status vmb_cross_scan(const void* x, void* xs, int B, int D, int H, int W, vmb_dtype dtype,
                          cudaStream_t stream);

/*
 * vmb_cross_merge - SS2D cross-merge (App. A, "VMamba": merge the four
 * sequence sets back into the 2-D map).
 *   ys  [B, 4, D, L]       per-direction outputs
 *   out [B, D, H, W]       out[b,d,h,w] = (ys0[p0] + ys2[p2]) + (ys1[p1] + ys3[p3]),
 *                          p0 = h*W + w, p1 = w*H + h, p2 = L-1-p0, p3 = L-1-p1,
 *                          summed in fp32 in exactly this order.
 */
vmb_status vmb_cross_merge(const void* ys, void* out, int B, int D, int H, int W,
                           vmb_dtype dtype, cudaStream_t stream);

/*
 * vmb_scan_workspace_bytes - bytes of zero-initialised device workspace that
 * vmb_selective_scan_fwd (path VMB_PATH_FULL) or vmb_mean_scan_fwd
 * (VMB_PATH_MEAN) needs for this problem on the current device, under any
 * flags (the larger of the plans of the two Bbar forms, which differ in tile
 * shape and chunking).  Always >= 256 (the status header).  The workspace
 * holds the status word and the chunk-carry exchange of the L-chunked scans.
 *
 * The workspace must be zero-filled once before its first use (cudaMemset or
 * a zeros tensor); afterwards every call leaves it ready for the next one.
 * Returns 0 for invalid arguments.
 */
size_t vmb_scan_workspace_bytes(int path, int B, int K, int D, int N, int H, int W,
                                vmb_dtype dtype);

/*
 * vmb_scan_kernel_count - number of kernels one vmb_selective_scan_fwd
 * (VMB_PATH_FULL) or vmb_mean_scan_fwd (VMB_PATH_MEAN) call launches for this
 * problem on the current device: 1, or 3 for the L-chunked full scan that
 * resolves the chunk carry in launches of its own.  0 for an empty problem or
 * invalid arguments.  (vmb_mean_scan_merge_fwd launches the mean scan's
 * kernels plus one merge kernel.)  Bookkeeping for timing tools; the paper
 * has no counterpart.
 */
int vmb_scan_kernel_count(int path, int B, int K, int D, int N, int H, int W, vmb_dtype dtype);

/*
 * vmb_selective_scan_fwd - full-channel selective scan over K directions
 * (App. A: selection Eq. 6, discretisation Eq. 4, recurrence Eq. 3), with the
 * discretisation fused into the scan:
 *   c = k*D + d,  delta_t = softplus(delta[b,k,d,t] + delta_bias[c])
 *   h_n(-1) = 0,  h_n(t) = exp(delta_t A[c,n]) h_n(t-1) + Bbar_n(t) u[b,k,d,t]
 *   y[b,k,d,t] = sum_n Cs[b,k,n,t] h_n(t) + Dskip[c] u[b,k,d,t]
 *   u, delta, y [B, K, D, L] (dtype);  Bs, Cs [B, K, N, L] (dtype)
 *   A [K*D, N], Dskip [K*D], delta_bias [K*D] (fp32)
 *   flags: VMB_FLAG_SOFTPLUS | VMB_FLAG_B_ZOH
 *   workspace: >= vmb_scan_workspace_bytes(VMB_PATH_FULL, ...) bytes, 256-B
 *   aligned, zero-filled before first use.
 * Supports 1 <= N <= 16 (VMB_ERR_UNSUPPORTED above) and any K >= 1.
 */
vmb_status vmb_selective_scan_fwd(const void* u, const void* delta, const float* A, const void* Bs,
                                  const void* Cs, const float* Dskip, const float* delta_bias,
                                  void* y, int B, int K, int D, int N, int H, int W,
                                  unsigned flags, vmb_dtype dtype, void* workspace,
                                  size_t workspace_bytes, cudaStream_t stream);

/*
 * vmb_mean_scan_fwd - VMeanba channel-mean scan (Sec. 2.2, Eq. 9:
 * y = T^-1(Mamba(T(Abar, Bbar u, C)))), T the mean over the D channels of one
 * (batch, direction), T^-1 the broadcast back to every channel:
 *   Abar_n(t)    = (1/D) sum_d exp(delta_{d,t} A[c_d,n])      (mean after the exp)
 *   (Bbar u)_n(t)= (1/D) sum_d Bbar_{d,n}(t) u[b,k,d,t]
 *   h_n(t) = Abar_n(t) h_n(t-1) + (Bbar u)_n(t),  ybar(t) = sum_n Cs[b,k,n,t] h_n(t)
 *   y[b,k,d,t] = ybar(t) + Dskip[c] u[b,k,d,t]      (VMB_FLAG_SKIP_MEAN:
 *                ybar(t) + (1/D) sum_d Dskip[c_d] u[b,k,d,t])
 * Same arguments as vmb_selective_scan_fwd, plus
 *   ybar [B, K, L] fp32 device pointer, or NULL: optional copy of ybar.
 * The recurrence runs once per (b, k) instead of once per (b, k, d).
 * Returns VMB_ERR_UNSUPPORTED when D * L >= 2^31 (the kernel addresses one
 * (b, k) slab with 32-bit offsets).
 */
vmb_status vmb_mean_scan_fwd(const void* u, const void* delta, const float* A, const void* Bs,
                             const void* Cs, const float* Dskip, const float* delta_bias, void* y,
                             float* ybar, int B, int K, int D, int N, int H, int W, unsigned flags,
                             vmb_dtype dtype, void* workspace, size_t workspace_bytes,
                             cudaStream_t stream);

/*
 * vmb_mean_scan_grouped_fwd - grouped basis: the reduced input set I_basis of
 * Sec. 2.1 with a reduced channel dimension d = groups instead of VMeanba's
 * d = 1 (Eq. 8 counts 9BLd FLOPs for it).  The D channels of each direction
 * are split into `groups` consecutive groups of D/groups channels; T is the
 * mean over each group and T^-1 broadcasts each group's ybar to its channels:
 *   ybar[b,k,g,t] as in vmb_mean_scan_fwd over channels g*D/G .. (g+1)*D/G - 1,
 *   y[b,k,d,t] = ybar[b,k,d/(D/G),t] + Dskip[c] u[b,k,d,t] (VMB_FLAG_SKIP_MEAN:
 *   the mean of Dskip u over the group).
 * Same arguments as vmb_mean_scan_fwd plus `groups` (>= 1, divides D;
 * VMB_ERR_INVALID_ARG otherwise); ybar, if not NULL, is [B, K, groups, L]
 * fp32.  groups = 1 is vmb_mean_scan_fwd; groups = D gives the full scan's y.
 * workspace: >= vmb_scan_workspace_bytes(VMB_PATH_MEAN, B, K*groups,
 * D/groups, N, H, W, dtype) bytes (the grouped problem runs as K*groups
 * directions of D/groups channels).
 */
vmb_status vmb_mean_scan_grouped_fwd(const void* u, const void* delta, const float* A, const void* Bs,
                                     const void* Cs, const float* Dskip, const float* delta_bias,
                                     void* y, float* ybar, int B, int K, int D, int N, int H, int W,
                                     int groups, unsigned flags, vmb_dtype dtype, void* workspace,
                                     size_t workspace_bytes, cudaStream_t stream);

/*
 * vmb_mean_scan_merge_fwd - the channel-mean path of an SS2D block (Sec. 2.2,
 * Eq. 9, then the App. A cross-merge) with the broadcast T^-1 fused into the
 * merge, so the per-channel output y [B, 4, D, L] is never written:
 *   every direction's u at the position it merges into is the map itself,
 *   u_k[b,d,p_k(h,w)] = x[b,d,h,w], hence
 *   out[b,d,h,w] = (y0 + y2) + (y1 + y3),
 *   y_k = ybar_k[b, p_k] + Dskip[k*D+d] x[b,d,h,w]  (p_k as in vmb_cross_merge;
 *         VMB_FLAG_SKIP_MEAN: y_k = ybar_k[b, p_k] + the mean skip term of k)
 *   u (= vmb_cross_scan(x)), delta [B, 4, D, L], Bs, Cs [B, 4, N, L] (dtype);
 *   A [4*D, N], Dskip [4*D], delta_bias [4*D] (fp32);
 *   x, out [B, D, H, W] (dtype), out must not alias x;
 *   ybar [B, 4, L] fp32, required: receives ybar_k(t) (plus the broadcast mean
 *   skip term under VMB_FLAG_SKIP_MEAN) and is read back by the merge.
 *   workspace: as vmb_mean_scan_fwd with K = 4 (VMB_PATH_MEAN).
 * The same fp32 operations in the same order as vmb_cross_merge applied to
 * vmb_mean_scan_fwd's y, so fp32 results are bit-identical to that unfused
 * pair; bf16 storage rounds once, at the end (the unfused pair rounds y
 * first).  Not in the paper as such: its kernels keep the steps apart.
 */
vmb_status vmb_mean_scan_merge_fwd(const void* u, const void* delta, const float* A, const void* Bs,
                                   const void* Cs, const float* Dskip, const float* delta_bias,
                                   const void* x, void* out, float* ybar, int B, int D, int N, int H,
                                   int W, unsigned flags, vmb_dtype dtype, void* workspace,
                                   size_t workspace_bytes, cudaStream_t stream);

/*
 * vmb_ss2d_full_fwd - the scan side of a full-channel SS2D block in one call
 * (App. A: cross-scan, the selective scan of Eqs. 3, 4 and 6, cross-merge)
 * without the cross-scanned sequences xs [B, 4, D, L] being written:
 *   y   = vmb_selective_scan_fwd(vmb_cross_scan(x), delta, ...) with K = 4,
 *   out = vmb_cross_merge(y)
 *   x, out [B, D, H, W] (dtype); y [B, 4, D, L] (dtype), written (the
 *   per-direction output); xt [B, D, W, H] (dtype), caller-owned scratch
 *   (overwritten); none of x, xt, y, out may alias another;
 *   delta [B, 4, D, L], Bs, Cs [B, 4, N, L] (dtype); A [4*D, N], Dskip [4*D],
 *   delta_bias [4*D] (fp32); flags and workspace as vmb_selective_scan_fwd with
 *   K = 4 (vmb_scan_workspace_bytes(VMB_PATH_FULL, B, 4, D, N, H, W, dtype)).
 * Where the warp-specialised scan kernel runs (16 states, rows of 16-byte
 * multiples, 16-byte aligned tensors, enough channel rows) direction k's step
 * l reads the value the cross-scan would have put there: directions 0 and 2
 * the (b, d) planes of x row by row (forward and reversed), directions 1 and 3
 * the rows of xt, the transpose of every plane (written by this call), so the
 * map moves 2 B*D*L elements instead of the cross-scan's 5 B*D*L.  Otherwise
 * the cross-scan is written into y and the scan runs in place.  Either way
 * the values and operations are those of the three separate calls, so y and
 * out are bit-identical to them.  Not in the paper as such: its kernels keep
 * the steps apart.
 */
vmb_status vmb_ss2d_full_fwd(const void* x, void* xt, const void* delta, const float* A,
                             const void* Bs, const void* Cs, const float* Dskip,
                             const float* delta_bias, void* y, void* out, int B, int D, int N,
                             int H, int W, unsigned flags, vmb_dtype dtype, void* workspace,
                             size_t workspace_bytes, cudaStream_t stream);

/*
 * vmb_ss2d_mean_fwd - the scan side of a VMeanba SS2D block in one call: the
 * App. A cross-scan, the channel-mean scan (Sec. 2.2, Eq. 9) and the App. A
 * cross-merge, without the cross-scanned sequences xs [B, 4, D, L] or the
 * per-channel output y ever being written.  Direction k's step l reads the
 * value the cross-scan would have put there: directions 0 and 2 read the
 * (b, d) planes of x row by row (forward and reversed), directions 1 and 3 the
 * rows of xt, the transpose of every plane (xt[b,d,w,h] = x[b,d,h,w], written
 * by this call); the merge applies the broadcast and the skip term:
 *   out = vmb_mean_scan_merge_fwd(vmb_cross_scan(x), delta, ..., x)
 *   x, out [B, D, H, W] (dtype), out must not alias x;
 *   xt [B, D, W, H] (dtype), caller-owned scratch (overwritten), aliasing
 *   neither x nor out;
 *   delta [B, 4, D, L], Bs, Cs [B, 4, N, L] (dtype); A [4*D, N], Dskip [4*D],
 *   delta_bias [4*D] (fp32); ybar [B, 4, L] fp32, required (as in
 *   vmb_mean_scan_merge_fwd); flags and workspace as vmb_mean_scan_fwd with
 *   K = 4 (vmb_scan_workspace_bytes(VMB_PATH_MEAN, B, 4, D, N, H, W, dtype)).
 * Moves 2 B*D*L elements for the map instead of the cross-scan's 5 B*D*L.
 * The same fp32 operations in the same order as that pair of calls, so fp32
 * results are bit-identical to it.  Not in the paper as such: its kernels keep
 * the steps apart.
 */
vmb_status vmb_ss2d_mean_fwd(const void* x, void* xt, const void* delta, const float* A,
                             const void* Bs, const void* Cs, const float* Dskip,
                             const float* delta_bias, void* out, float* ybar, int B, int D, int N,
                             int H, int W, unsigned flags, vmb_dtype dtype, void* workspace,
                             size_t workspace_bytes, cudaStream_t stream);

/*
 * vmb_selective_scan_fwd_noalloc - vmb_selective_scan_fwd for callers that
 * cannot allocate device memory (for example plugin code inside a framework
 * whose memory pool owns the device and forbids allocations of its own, or a
 * serving loop that must not allocate once it runs).  The paper has no
 * counterpart; this is a deployment convenience.
 *   Same arguments and results as vmb_selective_scan_fwd, without the
 *   workspace: the chunk-exchange scratch is a 16 MiB array built into the
 *   library, which every GPU that loads libvmb holds until the process exits.
 *   The call allocates nothing.
 *   Every argument check runs first: a rejected call queues nothing.
 *   Returns VMB_ERR_WORKSPACE when this call's plan (problem and flags) needs
 *   more than 16 MiB of scratch; vmb_scan_workspace_bytes(VMB_PATH_FULL, ...)
 *   <= 16 MiB guarantees that it does not.
 *   The first call made with a given device current looks up the array's
 *   device address on that device and keeps it for the life of the process;
 *   make that first call before any stream capture, and do not use this
 *   entry point across a cudaDeviceReset of that device.  Each call first
 *   clears the part of the array that must start at zero (an asynchronous
 *   memset on `stream`).  All calls share the one array per device, so calls
 *   that overlap in time on the GPU (other streams, other host threads) race
 *   and must be serialised by the caller.  Device-side wait timeouts have no
 *   readback for this entry point.
 */
vmb_status vmb_selective_scan_fwd_noalloc(const void* u, const void* delta, const float* A,
                                          const void* Bs, const void* Cs, const float* Dskip,
                                          const float* delta_bias, void* y, int B, int K, int D,
                                          int N, int H, int W, unsigned flags, vmb_dtype dtype,
                                          cudaStream_t stream);

/*
 * The paper's own kernel setting (Sec. 4, "Kernel Implementation"): the
 * discretisation runs outside the scan kernel, which reads the materialised
 * operands Abar and Bbar u.  These three calls reproduce that split, for
 * measuring it next to the fused scans above; they are not needed to compute
 * the SS2D output.  Operands are fp32; their sizes grow with N (a B=1 VMamba-T
 * stage-1 map with N = 16 materialises 2 x 154 MB).
 *
 * vmb_discretise_fwd - Eqs. 4 and 6 for every (b, k, d, n, l):
 *   delta = softplus(delta_raw + delta_bias[c]) (or raw + bias without
 *   VMB_FLAG_SOFTPLUS), dA[b,k,d,n,l] = exp(delta A[c,n]),
 *   dBu[b,k,d,n,l] = delta B[b,k,n,l] u[b,k,d,l] (Euler) or
 *   (exp(delta A) - 1) / A B u under VMB_FLAG_B_ZOH.
 *   u, delta [B,K,D,L], Bs [B,K,N,L] in dtype; A [K*D,N], delta_bias [K*D] fp32;
 *   dA, dBu [B,K,D,N,L] fp32 out.  flags: VMB_FLAG_SOFTPLUS | VMB_FLAG_B_ZOH.
 *   N in 1..16 (VMB_ERR_UNSUPPORTED above).
 *
 * vmb_discretise_mean_fwd - Eq. 9's T applied to the discretised operands:
 *   dAm[b,k,n,l] = mean_d exp(delta_d A[c_d,n]),
 *   dBum[b,k,n,l] = mean_d Bbar[b,k,d,n,l] u[b,k,d,l], fp32 [B,K,N,L] out (the
 *   [B,K,1,N,L] operands of the scan kernel).  Same inputs and flags as above.
 *
 * vmb_scan_only_fwd - Eq. 3 without the skip term on materialised operands of
 *   Dm channels per (b, k) (Dm = D for the full path, 1 after the mean):
 *   h[n] = dA h[n] + dBu from h = 0, y[b,k,d,l] = sum_n Cs[b,k,n,l] h[n].
 *   dA, dBu [B,K,Dm,N,L] fp32, Cs [B,K,N,L] in dtype, y [B,K,Dm,L] fp32 out.
 *   Deterministic; no workspace.  N in 1..16.
 */
vmb_status vmb_discretise_fwd(const void* u, const void* delta, const float* A, const void* Bs,
                              const float* delta_bias, float* dA, float* dBu, int B, int K, int D,
                              int N, int H, int W, unsigned flags, vmb_dtype dtype,
                              cudaStream_t stream);
vmb_status vmb_discretise_mean_fwd(const void* u, const void* delta, const float* A, const void* Bs,
                                   const float* delta_bias, float* dAm, float* dBum, int B, int K,
                                   int D, int N, int H, int W, unsigned flags, vmb_dtype dtype,
                                   cudaStream_t stream);
vmb_status vmb_scan_only_fwd(const float* dA, const float* dBu, const void* Cs, float* y, int B,
                             int K, int Dm, int N, int H, int W, vmb_dtype dtype,
                             cudaStream_t stream);

/*
 * vmb_selection_fwd - the selection functions of Eq. 6 (App. A): B, C and the
 * raw Delta of every step as linear maps of the scan input over the D channels
 * of that step and direction, with per-direction weights:
 *   Bs[b,k,n,l] = sum_d WB[k,n,d] u[b,k,d,l]      s_B = Linear_N(u)
 *   Cs[b,k,n,l] = sum_d WC[k,n,d] u[b,k,d,l]      s_C = Linear_N(u)
 *   z_r = sum_d Wz[k,r,d] u[b,k,d,l],  delta_raw[b,k,d,l] = sum_r Wup[k,d,r] z_r
 * The Delta branch is a rank-R map; R = 1 with Wup = 1 is the printed
 * s_Delta = Broadcast_D(Linear_1(u)).  The scans then apply
 * Delta = softplus(delta_raw + delta_bias) (VMB_FLAG_SOFTPLUS).
 *   u [B,K,D,L] (dtype); WB, WC [K,N,D], Wz [K,R,D], Wup [K,D,R] fp32;
 *   Bs, Cs [B,K,N,L], delta_raw [B,K,D,L] (dtype) out.  N and R in 1..16
 *   (VMB_ERR_UNSUPPORTED above).  Accumulation in fp32 (channels in order).
 */
vmb_status vmb_selection_fwd(const void* u, const float* WB, const float* WC, const float* Wz,
                             const float* Wup, void* Bs, void* Cs, void* delta_raw, int B, int K,
                             int D, int N, int R, int H, int W, vmb_dtype dtype, cudaStream_t stream);

/*
 * The selection functions with the Delta branch left in its low-rank form
 * (Eq. 6, App. A: s_Delta = Linear_D(Linear_R(u))), so the raw Deltas
 * [B,K,D,L] are never written: the scan expands them itself.
 *
 * vmb_selection_lowrank_fwd - as vmb_selection_fwd, but writes the rank-R
 *   intermediate z[b,k,r,l] = sum_d Wz[k,r,d] u[b,k,d,l] (fp32 [B,K,R,L],
 *   4-byte aligned) instead of delta_raw; no Wup.  Bs, Cs as there.
 *
 * vmb_selective_scan_lowrank_fwd - vmb_selective_scan_fwd with
 *   delta_raw[b,k,d,l] = sum_r Wup[k,d,r] z[b,k,r,l] (r in order, fp32)
 *   formed inside the scan from z [B,K,R,L] fp32 and Wup [K,D,R] fp32 (R in
 *   1..16; VMB_ERR_UNSUPPORTED above); every other argument, flag and the
 *   workspace (vmb_scan_workspace_bytes(VMB_PATH_FULL, ...)) as there; y must
 *   not alias u.  The warp-specialised scan (16 states, rows of 16-byte
 *   multiples, 16-byte aligned tensors, enough channel rows, Euler Bbar) reads
 *   z instead of the raw Deltas, i.e. R instead of D values per step and
 *   direction; for other plans the raw Deltas are written into y (rounded to
 *   the storage type) and the scan runs in place.  In fp32 the result is
 *   bit-identical to vmb_selection_fwd's raw Deltas fed to
 *   vmb_selective_scan_fwd; with bf16 storage the warp-specialised scan keeps
 *   the raw Deltas in fp32 (that pair rounds them to bf16 first).
 */
vmb_status vmb_selection_lowrank_fwd(const void* u, const float* WB, const float* WC, const float* Wz,
                                     void* Bs, void* Cs, float* z, int B, int K, int D, int N, int R, int H,
                                     int W, vmb_dtype dtype, cudaStream_t stream);
vmb_status vmb_selective_scan_lowrank_fwd(const void* u, const float* z, const float* Wup, const float* A,
                                          const void* Bs, const void* Cs, const float* Dskip,
                                          const float* delta_bias, void* y, int B, int K, int D, int N,
                                          int R, int H, int W, unsigned flags, vmb_dtype dtype,
                                          void* workspace, size_t workspace_bytes, cudaStream_t stream);

/*
 * vmb_mean_scan_lowrank_fwd - vmb_mean_scan_fwd (the channel-mean scan of
 *   Sec. 2.2, Eq. 9) with delta_raw = Wup z formed inside the scan, as in
 *   vmb_selective_scan_lowrank_fwd: z [B,K,R,L] fp32, Wup [K,D,R] fp32, R in
 *   1..16; every other argument (ybar optional), flag and the workspace
 *   (vmb_scan_workspace_bytes(VMB_PATH_MEAN, ...)) as vmb_mean_scan_fwd; y
 *   must not alias u.  For ranks up to 8 with the Euler Bbar each thread of
 *   the reduction forms the raw Delta of its step and channel (R FMAs) instead
 *   of reading it; otherwise the raw Deltas are written into y (rounded to the
 *   storage type) and the scan runs in place.  In fp32 the result is
 *   bit-identical to vmb_selection_fwd's raw Deltas fed to vmb_mean_scan_fwd.
 */
vmb_status vmb_mean_scan_lowrank_fwd(const void* u, const float* z, const float* Wup, const float* A,
                                     const void* Bs, const void* Cs, const float* Dskip,
                                     const float* delta_bias, void* y, float* ybar, int B, int K, int D,
                                     int N, int R, int H, int W, unsigned flags, vmb_dtype dtype,
                                     void* workspace, size_t workspace_bytes, cudaStream_t stream);

/*
 * vmb_mean_scan_train_fwd - vmb_mean_scan_grouped_fwd (groups = 1: the
 * channel-mean scan of Eq. 9) that also keeps, for vmb_mean_scan_bwd, the
 * group means it forms on the way:
 *   saved [B, K, groups, N + 1, L] fp32 out: rows n < N are Abar_n(t) (the
 *   mean of exp(delta A) over the group), row N is the mean of delta u.
 * The backward then skips recomputing them (N exponentials per element).
 * Same arguments and workspace as vmb_mean_scan_grouped_fwd plus `saved`
 * (not NULL, 4-byte aligned, 16-byte aligned for the backward's vector
 * loads); flags: VMB_FLAG_SOFTPLUS only (the backward covers Euler Bbar and
 * the per-channel skip term: VMB_FLAG_B_ZOH and VMB_FLAG_SKIP_MEAN give
 * VMB_ERR_UNSUPPORTED).  y and ybar are the grouped forward's, bit for bit.
 */
vmb_status vmb_mean_scan_train_fwd(const void* u, const void* delta, const float* A, const void* Bs,
                                   const void* Cs, const float* Dskip, const float* delta_bias,
                                   void* y, float* ybar, float* saved, int B, int K, int D, int N,
                                   int H, int W, int groups, unsigned flags, vmb_dtype dtype,
                                   void* workspace, size_t workspace_bytes, cudaStream_t stream);

/*
 * vmb_mean_scan_bwd - gradients of the channel-mean scan (Sec. 2.2, Eq. 9) or,
 * with groups > 1, of the grouped basis (Sec. 2.1, Eq. 8; vmb_mean_scan_grouped_fwd),
 * for the Euler Bbar and the per-channel skip term: the reverse-mode
 * derivative of the forward, given gy = dLoss/dy [B, K, D, L] (dtype).  Per
 * sequence (b, k, group) the states are recomputed forward, the adjoint
 *   lam_n(t) = C_n(t) sum_d gy_d(t) + Abar_n(t+1) lam_n(t+1)
 * runs backward in time, and the chain rule goes through the group mean and
 * the softplus.  Outputs (every one written, none accumulated into):
 *   gu, gdelta [B, K, D, L] (dtype): d/du and d/d(raw delta);
 *   gA [K*D, N], gDskip [K*D], gdelta_bias [K*D] (fp32), summed over the batch;
 *   gBs, gCs [B, K, N, L] (dtype), summed over the groups of each (b, k).
 * Same inputs as vmb_mean_scan_grouped_fwd (delta is the raw Delta); flags:
 * VMB_FLAG_SOFTPLUS (VMB_FLAG_B_ZOH and VMB_FLAG_SKIP_MEAN: VMB_ERR_UNSUPPORTED).
 * saved: the means vmb_mean_scan_train_fwd wrote for the same inputs,
 * groups and flags (4-byte aligned), or NULL to recompute them here.
 * workspace: >= vmb_mean_scan_bwd_workspace_bytes(...) bytes, 256-B aligned,
 * any contents (the group means, chunk carries and adjoints of every
 * sequence, fp32: about 2 x (N + 2) x 4 bytes per (b, k, group, step)).  Every
 * reduction runs in a fixed order: results are deterministic.  The paper
 * trains no VMeanba layer (it replaces layers of a trained model); this is the
 * chain rule of the forward defined there.
 */
vmb_status vmb_mean_scan_bwd(const void* u, const void* delta, const float* A, const void* Bs,
                             const void* Cs, const float* Dskip, const float* delta_bias,
                             const void* gy, const float* saved, void* gu, void* gdelta, float* gA,
                             void* gBs, void* gCs, float* gDskip, float* gdelta_bias, int B, int K,
                             int D, int N, int H, int W, int groups, unsigned flags,
                             vmb_dtype dtype, void* workspace, size_t workspace_bytes,
                             cudaStream_t stream);
size_t vmb_mean_scan_bwd_workspace_bytes(int B, int K, int D, int N, int H, int W, int groups,
                                         vmb_dtype dtype);

/*
 * vmb_read_status - synchronise `stream`, then return and clear the device
 * error word of `workspace` (VMB_OK, VMB_ERR_TIMEOUT or VMB_ERR_BOUNDS).  A
 * device-side error leaves the outputs of that call undefined but the CUDA
 * context usable.  Returns VMB_ERR_CUDA if the synchronisation fails.
 */
vmb_status vmb_read_status(void* workspace, cudaStream_t stream);

/* Static description of a status code (never NULL). */
const char* vmb_status_string(vmb_status status);

/* Library version: major*10000 + minor*100 + patch. */
int vmb_version(void);

#ifdef __cplusplus
}
#endif

#endif /* VMB_H */
