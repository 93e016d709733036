// vmb_abi.cu - the extern "C" entry points of libvmb (declared in include/vmb.h):
// argument validation, plan and workspace sizing, launch on the caller's stream.
#include <limits.h>

#include <atomic>
#include <mutex>

#include "vmb_common.cuh"
#include "vmb_internal.h"
#include "vmb_testing.h"

namespace vmb {

namespace {
std::atomic<int> g_force_shape{-1}, g_force_chunks{0}, g_force_tc{0};
}  // namespace

int forced_full_shape(int* chunks) {
    *chunks = g_force_chunks.load(std::memory_order_relaxed);
    return g_force_shape.load(std::memory_order_relaxed);
}
int forced_mean_chunk() { return g_force_tc.load(std::memory_order_relaxed); }

int device_sm_count() {
    static std::mutex mu;
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    std::lock_guard<std::mutex> g(mu);
    if (dev >= 0 && dev < 64 && cache[dev] > 0) return cache[dev];
    int n = 1;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) n = 1;
    if (dev >= 0 && dev < 64) cache[dev] = n;
    return n;
}

namespace {

bool mul_ok(long long a, long long b, long long* out) {
    if (a < 0 || b < 0) return false;
    if (a != 0 && b > LLONG_MAX / a) return false;
    *out = a * b;
    return true;
}

bool count(long long* out, std::initializer_list<long long> dims) {
    long long v = 1;
    for (long long d : dims)
        if (!mul_ok(v, d, &v)) return false;
    *out = v;
    return true;
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

size_t esize(vmb_dtype dt) { return dt == VMB_BF16 ? 2 : 4; }

bool dtype_ok(vmb_dtype dt) { return dt == VMB_F32 || dt == VMB_BF16; }

constexpr unsigned kKnownFlags =
    VMB_FLAG_SOFTPLUS | VMB_FLAG_B_ZOH | VMB_FLAG_SKIP_MEAN | VMB_FLAG_TEST_SUPPRESS_PUBLISH;

// Shared checks of the cross-scan / cross-merge calls.  *empty is set for a
// problem with no elements.
vmb_status check_csm(const void* in, const void* out, int B, int D, int H, int W, vmb_dtype dt, bool* empty) {
    if (!dtype_ok(dt) || B < 0 || D < 0 || H < 0 || W < 0) return VMB_ERR_INVALID_ARG;
    long long n4 = 0;
    if (!count(&n4, {B, 4, D, H, W})) return VMB_ERR_INVALID_ARG;
    *empty = n4 == 0;
    if (*empty) return VMB_OK;
    if ((long long)H * W > INT_MAX) return VMB_ERR_UNSUPPORTED;
    if (!in || !out) return VMB_ERR_INVALID_ARG;
    if (!aligned(in, esize(dt)) || !aligned(out, esize(dt))) return VMB_ERR_MISALIGNED;
    return VMB_OK;
}

vmb_status check_scan(const ScanArgs& a, bool mean, bool* empty) {
    if (!dtype_ok(a.dtype)) return VMB_ERR_INVALID_ARG;
    if (a.B < 0 || a.K < 0 || a.D < 0 || a.N < 0 || a.L < 0) return VMB_ERR_INVALID_ARG;
    if (a.flags & ~kKnownFlags) return VMB_ERR_INVALID_ARG;
    if (!mean && (a.flags & VMB_FLAG_SKIP_MEAN)) return VMB_ERR_INVALID_ARG;
    long long n = 0, nbc = 0;
    if (!count(&n, {a.B, a.K, a.D, a.L}) || !count(&nbc, {a.B, a.K, a.N > 0 ? a.N : 1, a.L}))
        return VMB_ERR_INVALID_ARG;
    *empty = n == 0;
    if (*empty) return VMB_OK;
    if (a.N < 1) return VMB_ERR_INVALID_ARG;
    if (a.N > 16) return VMB_ERR_UNSUPPORTED;
    long long grid_rows = 0;
    if (!count(&grid_rows, {a.B, a.K, a.D}) || grid_rows > INT_MAX / 2) return VMB_ERR_UNSUPPORTED;
    if (!a.u || !a.delta || !a.A || !a.Bs || !a.Cs || !a.Dskip || !a.bias || (!a.y && !a.no_bcast))
        return VMB_ERR_INVALID_ARG;
    if (a.no_bcast && !a.ybar) return VMB_ERR_INVALID_ARG;
    const size_t es = esize(a.dtype);
    if (!aligned(a.u, es) || !aligned(a.delta, es) || !aligned(a.Bs, es) || !aligned(a.Cs, es) ||
        (a.y && !aligned(a.y, es)) || !aligned(a.A, 4) || !aligned(a.Dskip, 4) || !aligned(a.bias, 4) ||
        (a.ybar && !aligned(a.ybar, 4)))
        return VMB_ERR_MISALIGNED;
    return VMB_OK;
}

// Checks of the discretisation calls; sets a.L.
vmb_status check_disc(DiscArgs& a, int H, int W, bool mean, bool* empty) {
    if (!dtype_ok(a.dtype) || a.B < 0 || a.K < 0 || a.D < 0 || a.N < 0 || H < 0 || W < 0) return VMB_ERR_INVALID_ARG;
    if (a.flags & ~(VMB_FLAG_SOFTPLUS | VMB_FLAG_B_ZOH)) return VMB_ERR_INVALID_ARG;
    long long n = 0, nop = 0;
    if (!count(&n, {a.B, a.K, a.D, H, W}) || !count(&nop, {a.B, a.K, mean ? 1 : a.D, a.N > 0 ? a.N : 1, H, W}))
        return VMB_ERR_INVALID_ARG;
    *empty = n == 0;
    if (*empty) return VMB_OK;
    if ((long long)H * W > INT_MAX) return VMB_ERR_UNSUPPORTED;
    a.L = H * W;
    if (a.N < 1) return VMB_ERR_INVALID_ARG;
    if (a.N > 16) return VMB_ERR_UNSUPPORTED;
    long long rows = 0;
    if (!count(&rows, {a.B, a.K, a.D}) || rows > INT_MAX / 2) return VMB_ERR_UNSUPPORTED;
    if (!a.u || !a.delta || !a.A || !a.Bs || !a.bias || !a.dA || !a.dBu) return VMB_ERR_INVALID_ARG;
    const size_t es = esize(a.dtype);
    if (!aligned(a.u, es) || !aligned(a.delta, es) || !aligned(a.Bs, es) || !aligned(a.A, 4) || !aligned(a.bias, 4) ||
        !aligned(a.dA, 4) || !aligned(a.dBu, 4))
        return VMB_ERR_MISALIGNED;
    return VMB_OK;
}

vmb_status run_scan(ScanArgs& a, bool mean, cudaStream_t stream) {
    bool empty = false;
    vmb_status s = check_scan(a, mean, &empty);
    if (s != VMB_OK || empty) return s;
    if (!a.ws) return VMB_ERR_WORKSPACE;
    if (!aligned(a.ws, 256)) return VMB_ERR_MISALIGNED;
    ScanPlan plan{};
    s = mean ? plan_mean(a, &plan) : plan_full(a, &plan);
    if (s != VMB_OK) return s;
    if (a.ws_bytes < plan.ws_bytes) return VMB_ERR_WORKSPACE;
    return mean ? launch_mean(a, plan, stream) : launch_full(a, plan, stream);
}

// Workspace bytes of the plans for each of `flag_sets` (the largest).
size_t plan_bytes(int path, const unsigned* flag_sets, int nsets, int B, int K, int D, int N, int H, int W,
                  vmb_dtype dtype) {
    if (path != VMB_PATH_FULL && path != VMB_PATH_MEAN) return 0;
    if (H < 0 || W < 0 || (long long)H * W > INT_MAX) return 0;
    ScanArgs a{};
    a.B = B;
    a.K = K;
    a.D = D;
    a.N = N;
    a.L = H * W;
    a.dtype = dtype;
    // shape-only validation: stand-in non-null, aligned pointers
    static const float dummy[4] = {0, 0, 0, 0};
    a.u = a.delta = a.Bs = a.Cs = dummy;
    a.A = a.Dskip = a.bias = dummy;
    a.y = const_cast<float*>(dummy);
    size_t need = 0;
    for (int i = 0; i < nsets; ++i) {
        a.flags = flag_sets[i];
        bool empty = false;
        if (check_scan(a, path == VMB_PATH_MEAN, &empty) != VMB_OK) return 0;
        if (empty) return 256;
        ScanPlan plan{};
        if ((path == VMB_PATH_MEAN ? plan_mean(a, &plan) : plan_full(a, &plan)) != VMB_OK) return 0;
        if (plan.ws_bytes > need) need = plan.ws_bytes;
    }
    return need;
}
}  // namespace

vmb_status validate_scan(const ScanArgs& a, bool mean, bool* empty) { return check_scan(a, mean, empty); }

}  // namespace vmb

using namespace vmb;

extern "C" {

vmb_status vmb_cross_scan(const void* x, void* xs, int B, int D, int H, int W, vmb_dtype dtype, cudaStream_t stream) {
    bool empty = false;
    vmb_status s = check_csm(x, xs, B, D, H, W, dtype, &empty);
    if (s != VMB_OK || empty) return s;
    return launch_cross_scan(x, xs, B, D, H, W, dtype, stream);
}

vmb_status vmb_cross_merge(const void* ys, void* out, int B, int D, int H, int W, vmb_dtype dtype, cudaStream_t stream) {
    bool empty = false;
    vmb_status s = check_csm(ys, out, B, D, H, W, dtype, &empty);
    if (s != VMB_OK || empty) return s;
    return launch_cross_merge(ys, out, B, D, H, W, dtype, stream);
}

size_t vmb_scan_workspace_bytes(int path, int B, int K, int D, int N, int H, int W, vmb_dtype dtype) {
    // The planners pick the tile shape and chunk count from the problem and
    // the B-bar form (the zero-order-hold kernels have their own shapes), so
    // the query covers both forms: one workspace serves every flag setting.
    static const unsigned forms[2] = {0u, (unsigned)VMB_FLAG_B_ZOH};
    return plan_bytes(path, forms, 2, B, K, D, N, H, W, dtype);
}

size_t vmb_testing_plan_workspace_bytes(int path, unsigned flags, int B, int K, int D, int N, int H, int W,
                                        vmb_dtype dtype) {
    return plan_bytes(path, &flags, 1, B, K, D, N, H, W, dtype);
}

int vmb_scan_kernel_count(int path, int B, int K, int D, int N, int H, int W, vmb_dtype dtype) {
    if (path != VMB_PATH_FULL && path != VMB_PATH_MEAN) return 0;
    if (H < 0 || W < 0 || (long long)H * W > INT_MAX) return 0;
    ScanArgs a{};
    a.B = B;
    a.K = K;
    a.D = D;
    a.N = N;
    a.L = H * W;
    a.dtype = dtype;
    static const float dummy[4] = {0, 0, 0, 0};
    a.u = a.delta = a.Bs = a.Cs = dummy;
    a.A = a.Dskip = a.bias = dummy;
    a.y = const_cast<float*>(dummy);
    bool empty = false;
    if (check_scan(a, path == VMB_PATH_MEAN, &empty) != VMB_OK || empty) return 0;
    ScanPlan plan{};
    if (path == VMB_PATH_MEAN) return plan_mean(a, &plan) == VMB_OK ? 1 : 0;
    return plan_full(a, &plan) == VMB_OK ? full_plan_launches(plan) : 0;
}

vmb_status vmb_selective_scan_fwd(const void* u, const void* delta, const float* A, const void* Bs, const void* Cs,
                                  const float* Dskip, const float* delta_bias, void* y, int B, int K, int D, int N,
                                  int H, int W, unsigned flags, vmb_dtype dtype, void* workspace,
                                  size_t workspace_bytes, cudaStream_t stream) {
    if (H < 0 || W < 0) return VMB_ERR_INVALID_ARG;
    if ((long long)H * W > INT_MAX) return VMB_ERR_UNSUPPORTED;
    ScanArgs a{u, delta, A, Bs, Cs, Dskip, delta_bias, y, nullptr, B, K, D, N, H * W, flags, dtype, workspace, workspace_bytes};
    return run_scan(a, false, stream);
}

vmb_status vmb_mean_scan_fwd(const void* u, const void* delta, const float* A, const void* Bs, const void* Cs,
                             const float* Dskip, const float* delta_bias, void* y, float* ybar, int B, int K, int D,
                             int N, int H, int W, unsigned flags, vmb_dtype dtype, void* workspace,
                             size_t workspace_bytes, cudaStream_t stream) {
    if (H < 0 || W < 0) return VMB_ERR_INVALID_ARG;
    if ((long long)H * W > INT_MAX) return VMB_ERR_UNSUPPORTED;
    ScanArgs a{u, delta, A, Bs, Cs, Dskip, delta_bias, y, ybar, B, K, D, N, H * W, flags, dtype, workspace, workspace_bytes};
    return run_scan(a, true, stream);
}

vmb_status vmb_mean_scan_grouped_fwd(const void* u, const void* delta, const float* A, const void* Bs, const void* Cs,
                                     const float* Dskip, const float* delta_bias, void* y, float* ybar, int B, int K,
                                     int D, int N, int H, int W, int groups, unsigned flags, vmb_dtype dtype,
                                     void* workspace, size_t workspace_bytes, cudaStream_t stream) {
    if (H < 0 || W < 0 || groups < 1) return VMB_ERR_INVALID_ARG;
    if (D % groups != 0) return VMB_ERR_INVALID_ARG;
    if ((long long)H * W > INT_MAX) return VMB_ERR_UNSUPPORTED;
    long long kg = 0;
    if (!count(&kg, {K, groups}) || kg > INT_MAX) return VMB_ERR_UNSUPPORTED;
    // the (b, k, g) sequences are the (b, k') sequences of a problem with K*G
    // directions of D/G channels: u, delta, y rows, A, bias, Dskip and ybar
    // are laid out identically; only B / C rows are shared by G sequences
    ScanArgs a{u, delta, A, Bs, Cs, Dskip, delta_bias, y, ybar, B, (int)kg, D / groups, N, H * W, flags, dtype,
               workspace, workspace_bytes};
    a.bc_group = groups;
    return run_scan(a, true, stream);
}

vmb_status vmb_mean_scan_train_fwd(const void* u, const void* delta, const float* A, const void* Bs, const void* Cs,
                                   const float* Dskip, const float* delta_bias, void* y, float* ybar, float* saved,
                                   int B, int K, int D, int N, int H, int W, int groups, unsigned flags,
                                   vmb_dtype dtype, void* workspace, size_t workspace_bytes, cudaStream_t stream) {
    if (H < 0 || W < 0 || groups < 1) return VMB_ERR_INVALID_ARG;
    if (D % groups != 0) return VMB_ERR_INVALID_ARG;
    if ((long long)H * W > INT_MAX) return VMB_ERR_UNSUPPORTED;
    if (flags & (VMB_FLAG_B_ZOH | VMB_FLAG_SKIP_MEAN)) {
        // the backward covers Euler Bbar and the per-channel skip term; anything
        // else is rejected after the shape checks the other entry points make
        if (!dtype_ok(dtype) || B < 0 || K < 0 || D < 0 || N < 0) return VMB_ERR_INVALID_ARG;
        return VMB_ERR_UNSUPPORTED;
    }
    long long kg = 0;
    if (!count(&kg, {K, groups}) || kg > INT_MAX) return VMB_ERR_UNSUPPORTED;
    ScanArgs a{u, delta, A, Bs, Cs, Dskip, delta_bias, y, ybar, B, (int)kg, D / groups, N, H * W, flags, dtype,
               workspace, workspace_bytes};
    a.bc_group = groups;
    bool empty = false;
    vmb_status s = validate_scan(a, true, &empty);
    if (s != VMB_OK || empty) return s;
    if (!saved) return VMB_ERR_INVALID_ARG;
    if (!aligned(saved, 4)) return VMB_ERR_MISALIGNED;
    a.saved = saved;
    return run_scan(a, true, stream);
}

vmb_status vmb_mean_scan_merge_fwd(const void* u, const void* delta, const float* A, const void* Bs, const void* Cs,
                                   const float* Dskip, const float* delta_bias, const void* x, void* out, float* ybar,
                                   int B, int D, int N, int H, int W, unsigned flags, vmb_dtype dtype, void* workspace,
                                   size_t workspace_bytes, cudaStream_t stream) {
    bool empty = false;
    vmb_status s = check_csm(x, out, B, D, H, W, dtype, &empty);
    if (s != VMB_OK || empty) return s;
    if (x == out) return VMB_ERR_INVALID_ARG;
    ScanArgs a{u, delta, A, Bs, Cs, Dskip, delta_bias, nullptr, ybar, B, 4, D, N, H * W, flags, dtype,
               workspace, workspace_bytes};
    a.no_bcast = true;
    s = run_scan(a, true, stream);
    if (s != VMB_OK) return s;
    return launch_mean_merge(x, ybar, Dskip, out, B, D, H, W, (flags & VMB_FLAG_SKIP_MEAN) == 0, dtype, stream);
}

vmb_status vmb_ss2d_mean_fwd(const void* x, void* xt, const void* delta, const float* A, const void* Bs,
                             const void* Cs, const float* Dskip, const float* delta_bias, void* out, float* ybar,
                             int B, int D, int N, int H, int W, unsigned flags, vmb_dtype dtype, void* workspace,
                             size_t workspace_bytes, cudaStream_t stream) {
    bool empty = false;
    vmb_status s = check_csm(x, out, B, D, H, W, dtype, &empty);
    if (s != VMB_OK || empty) return s;
    if (x == out || !xt || xt == x || xt == out) return VMB_ERR_INVALID_ARG;
    if (!aligned(xt, esize(dtype))) return VMB_ERR_MISALIGNED;
    // the channel-mean scan reads each direction's steps straight from the map
    // (rows of x) or its transpose (rows of xt), with no materialised
    // cross-scan; it stops at ybar, and the merge applies the broadcast and the
    // skip term
    ScanArgs a{x, delta, A, Bs, Cs, Dskip, delta_bias, nullptr, ybar, B, 4, D, N, H * W, flags, dtype,
               workspace, workspace_bytes};
    a.no_bcast = true;
    a.gather_h = H;
    a.u_t = xt;
    // every check (arguments, plan, workspace size) before the first launch
    bool scan_empty = false;
    s = check_scan(a, true, &scan_empty);
    if (s != VMB_OK) return s;
    if (!workspace) return VMB_ERR_WORKSPACE;
    if (!aligned(workspace, 256)) return VMB_ERR_MISALIGNED;
    ScanPlan plan{};
    s = plan_mean(a, &plan);
    if (s != VMB_OK) return s;
    if (workspace_bytes < plan.ws_bytes) return VMB_ERR_WORKSPACE;
    s = launch_map_transpose(x, xt, B, D, H, W, dtype, stream);
    if (s != VMB_OK) return s;
    s = launch_mean(a, plan, stream);
    if (s != VMB_OK) return s;
    return launch_mean_merge(x, ybar, Dskip, out, B, D, H, W, (flags & VMB_FLAG_SKIP_MEAN) == 0, dtype, stream);
}

vmb_status vmb_selective_scan_lowrank_fwd(const void* u, const float* z, const float* Wup, const float* A,
                                          const void* Bs, const void* Cs, const float* Dskip, const float* delta_bias,
                                          void* y, int B, int K, int D, int N, int R, int H, int W, unsigned flags,
                                          vmb_dtype dtype, void* workspace, size_t workspace_bytes, cudaStream_t stream) {
    if (H < 0 || W < 0 || R < 0) return VMB_ERR_INVALID_ARG;
    if ((long long)H * W > INT_MAX) return VMB_ERR_UNSUPPORTED;
    ScanArgs a{u, z, A, Bs, Cs, Dskip, delta_bias, y, nullptr, B, K, D, N, H * W, flags, dtype, workspace,
               workspace_bytes};
    a.Wup = Wup;
    a.R = R;
    bool empty = false;
    vmb_status s = check_scan(a, false, &empty);
    if (s != VMB_OK || empty) return s;
    if (R < 1) return VMB_ERR_INVALID_ARG;
    if (R > 16) return VMB_ERR_UNSUPPORTED;
    if (!Wup || u == y) return VMB_ERR_INVALID_ARG;
    if (!aligned(z, 4) || !aligned(Wup, 4)) return VMB_ERR_MISALIGNED;
    if (!workspace) return VMB_ERR_WORKSPACE;
    if (!aligned(workspace, 256)) return VMB_ERR_MISALIGNED;
    ScanPlan plan{};
    s = plan_full(a, &plan);
    if (s != VMB_OK) return s;
    if (workspace_bytes < plan.ws_bytes) return VMB_ERR_WORKSPACE;
    if (full_plan_gathers(plan)) return launch_full(a, plan, stream);
    // a plan whose kernel reads materialised raw Deltas: they are written into
    // y and the scan runs in place (each of its CTAs reads the steps of its own
    // rows before it writes them, and no other CTA touches them)
    ScanArgs m = a;
    m.delta = y;
    m.Wup = nullptr;
    m.R = 0;
    ScanPlan mplan{};
    s = plan_full(m, &mplan);
    if (s != VMB_OK) return s;
    if (workspace_bytes < mplan.ws_bytes) return VMB_ERR_WORKSPACE;
    s = launch_lowrank_expand(z, Wup, y, B, K, D, R, H * W, dtype, stream);
    if (s != VMB_OK) return s;
    return launch_full(m, mplan, stream);
}

vmb_status vmb_mean_scan_lowrank_fwd(const void* u, const float* z, const float* Wup, const float* A,
                                     const void* Bs, const void* Cs, const float* Dskip, const float* delta_bias,
                                     void* y, float* ybar, int B, int K, int D, int N, int R, int H, int W,
                                     unsigned flags, vmb_dtype dtype, void* workspace, size_t workspace_bytes,
                                     cudaStream_t stream) {
    if (H < 0 || W < 0 || R < 0) return VMB_ERR_INVALID_ARG;
    if ((long long)H * W > INT_MAX) return VMB_ERR_UNSUPPORTED;
    ScanArgs a{u, z, A, Bs, Cs, Dskip, delta_bias, y, ybar, B, K, D, N, H * W, flags, dtype, workspace,
               workspace_bytes};
    a.Wup = Wup;
    a.R = R;
    bool empty = false;
    vmb_status s = check_scan(a, true, &empty);
    if (s != VMB_OK || empty) return s;
    if (R < 1) return VMB_ERR_INVALID_ARG;
    if (R > 16) return VMB_ERR_UNSUPPORTED;
    if (!Wup || u == y) return VMB_ERR_INVALID_ARG;
    if (!aligned(z, 4) || !aligned(Wup, 4)) return VMB_ERR_MISALIGNED;
    if (!workspace) return VMB_ERR_WORKSPACE;
    if (!aligned(workspace, 256)) return VMB_ERR_MISALIGNED;
    ScanPlan plan{};
    s = plan_mean(a, &plan);
    if (s != VMB_OK) return s;
    if (workspace_bytes < plan.ws_bytes) return VMB_ERR_WORKSPACE;
    if (!(flags & VMB_FLAG_B_ZOH) && R <= 8) return launch_mean(a, plan, stream);
    // ranks above 8 and the ZOH form: the raw Deltas are written into y and
    // the scan runs in place (a CTA reads the Deltas of its chunk before it
    // writes that chunk's y, and no other CTA touches them)
    ScanArgs m = a;
    m.delta = y;
    m.Wup = nullptr;
    m.R = 0;
    s = launch_lowrank_expand(z, Wup, y, B, K, D, R, H * W, dtype, stream);
    if (s != VMB_OK) return s;
    return launch_mean(m, plan, stream);
}

vmb_status vmb_ss2d_full_fwd(const void* x, void* xt, const void* delta, const float* A, const void* Bs,
                             const void* Cs, const float* Dskip, const float* delta_bias, void* y, void* out, int B,
                             int D, int N, int H, int W, unsigned flags, vmb_dtype dtype, void* workspace,
                             size_t workspace_bytes, cudaStream_t stream) {
    bool empty = false;
    vmb_status s = check_csm(x, out, B, D, H, W, dtype, &empty);
    if (s != VMB_OK || empty) return s;
    if (x == out || !xt || !y || xt == x || xt == out || xt == y || y == x || y == out) return VMB_ERR_INVALID_ARG;
    if (!aligned(xt, esize(dtype))) return VMB_ERR_MISALIGNED;
    // the full scan reads each direction's steps from the map (rows of x) or its
    // transpose (rows of xt), with no materialised cross-scan, and writes y;
    // the merge then sums the four directions
    ScanArgs a{x, delta, A, Bs, Cs, Dskip, delta_bias, y, nullptr, B, 4, D, N, H * W, flags, dtype,
               workspace, workspace_bytes};
    a.gather_h = H;
    a.u_t = xt;
    // every check (arguments, plan, workspace size) before the first launch
    bool scan_empty = false;
    s = check_scan(a, false, &scan_empty);
    if (s != VMB_OK) return s;
    if (!workspace) return VMB_ERR_WORKSPACE;
    if (!aligned(workspace, 256)) return VMB_ERR_MISALIGNED;
    ScanPlan plan{};
    s = plan_full(a, &plan);
    if (s != VMB_OK) return s;
    if (workspace_bytes < plan.ws_bytes) return VMB_ERR_WORKSPACE;
    if (full_plan_gathers(plan)) {
        s = launch_map_transpose(x, xt, B, D, H, W, dtype, stream);
        if (s != VMB_OK) return s;
        s = launch_full(a, plan, stream);
    } else {
        // a plan whose kernel reads materialised sequences: the cross-scan goes
        // into y and the scan runs in place (each of its CTAs reads the steps of
        // its own rows before it writes them, and no other CTA touches them)
        ScanArgs m = a;
        m.u = y;
        m.gather_h = 0;
        m.u_t = nullptr;
        ScanPlan mplan{};
        s = plan_full(m, &mplan);
        if (s != VMB_OK) return s;
        if (workspace_bytes < mplan.ws_bytes) return VMB_ERR_WORKSPACE;
        s = launch_cross_scan(x, y, B, D, H, W, dtype, stream);
        if (s != VMB_OK) return s;
        s = launch_full(m, mplan, stream);
    }
    if (s != VMB_OK) return s;
    return launch_cross_merge(y, out, B, D, H, W, dtype, stream);
}

// Checks of the backward call; sets *empty for a problem with no elements.
static vmb_status check_bwd(const MeanBwdArgs& a, bool* empty) {
    if (!dtype_ok(a.dtype) || a.B < 0 || a.K < 0 || a.D < 0 || a.N < 0 || a.L < 0) return VMB_ERR_INVALID_ARG;
    if (a.flags & ~(unsigned)(VMB_FLAG_SOFTPLUS | VMB_FLAG_B_ZOH | VMB_FLAG_SKIP_MEAN)) return VMB_ERR_INVALID_ARG;
    long long n = 0, nbc = 0;
    if (!count(&n, {a.B, a.K, a.D, a.L}) || !count(&nbc, {a.B, a.K, a.N > 0 ? a.N : 1, a.L}))
        return VMB_ERR_INVALID_ARG;
    *empty = n == 0;
    if (*empty) return VMB_OK;
    if (a.N < 1 || a.groups < 1 || a.D % a.groups != 0) return VMB_ERR_INVALID_ARG;
    if (a.N > 16) return VMB_ERR_UNSUPPORTED;
    if (a.flags & (VMB_FLAG_B_ZOH | VMB_FLAG_SKIP_MEAN)) return VMB_ERR_UNSUPPORTED;  // Euler Bbar, per-channel skip
    long long rows = 0;
    if (!count(&rows, {a.B, a.K, a.D}) || rows > INT_MAX / 2 || (long long)a.B * a.K * a.groups > INT_MAX / 16)
        return VMB_ERR_UNSUPPORTED;
    const void* ptrs[] = {a.u, a.delta, a.A, a.Bs, a.Cs, a.Dskip, a.bias, a.gy, a.gu, a.gdelta, a.gA, a.gBs, a.gCs,
                          a.gDskip, a.gbias};
    for (const void* q : ptrs)
        if (!q) return VMB_ERR_INVALID_ARG;
    if (a.saved && !aligned(a.saved, 4)) return VMB_ERR_MISALIGNED;
    const size_t es = esize(a.dtype);
    const void* elems[] = {a.u, a.delta, a.Bs, a.Cs, a.gy, a.gu, a.gdelta, a.gBs, a.gCs};
    for (const void* q : elems)
        if (!aligned(q, es)) return VMB_ERR_MISALIGNED;
    const void* params[] = {a.A, a.Dskip, a.bias, a.gA, a.gDskip, a.gbias};
    for (const void* q : params)
        if (!aligned(q, 4)) return VMB_ERR_MISALIGNED;
    return VMB_OK;
}

vmb_status vmb_discretise_fwd(const void* u, const void* delta, const float* A, const void* Bs,
                              const float* delta_bias, float* dA, float* dBu, int B, int K, int D, int N, int H,
                              int W, unsigned flags, vmb_dtype dtype, cudaStream_t stream) {
    DiscArgs a{u, delta, A, Bs, delta_bias, dA, dBu, B, K, D, N, 0, flags, dtype};
    bool empty = false;
    vmb_status s = check_disc(a, H, W, false, &empty);
    if (s != VMB_OK || empty) return s;
    return launch_discretise(a, false, stream);
}

vmb_status vmb_discretise_mean_fwd(const void* u, const void* delta, const float* A, const void* Bs,
                                   const float* delta_bias, float* dAm, float* dBum, int B, int K, int D, int N,
                                   int H, int W, unsigned flags, vmb_dtype dtype, cudaStream_t stream) {
    DiscArgs a{u, delta, A, Bs, delta_bias, dAm, dBum, B, K, D, N, 0, flags, dtype};
    bool empty = false;
    vmb_status s = check_disc(a, H, W, true, &empty);
    if (s != VMB_OK || empty) return s;
    return launch_discretise(a, true, stream);
}

vmb_status vmb_scan_only_fwd(const float* dA, const float* dBu, const void* Cs, float* y, int B, int K, int Dm,
                             int N, int H, int W, vmb_dtype dtype, cudaStream_t stream) {
    if (!dtype_ok(dtype) || B < 0 || K < 0 || Dm < 0 || N < 0 || H < 0 || W < 0) return VMB_ERR_INVALID_ARG;
    long long n = 0, nop = 0;
    if (!count(&n, {B, K, Dm, H, W}) || !count(&nop, {B, K, Dm, N > 0 ? N : 1, H, W})) return VMB_ERR_INVALID_ARG;
    if (n == 0) return VMB_OK;
    if ((long long)H * W > INT_MAX - 1024) return VMB_ERR_UNSUPPORTED;  // segment offsets stay in int
    if (N < 1) return VMB_ERR_INVALID_ARG;
    if (N > 16) return VMB_ERR_UNSUPPORTED;
    if (!dA || !dBu || !Cs || !y) return VMB_ERR_INVALID_ARG;
    if (!aligned(dA, 4) || !aligned(dBu, 4) || !aligned(y, 4) || !aligned(Cs, esize(dtype))) return VMB_ERR_MISALIGNED;
    OnlyArgs a{dA, dBu, Cs, y, B, K, Dm, N, H * W, dtype};
    return launch_scan_only(a, stream);
}

vmb_status vmb_selection_fwd(const void* u, const float* WB, const float* WC, const float* Wz, const float* Wup,
                             void* Bs, void* Cs, void* delta_raw, int B, int K, int D, int N, int R, int H, int W,
                             vmb_dtype dtype, cudaStream_t stream) {
    if (!dtype_ok(dtype) || B < 0 || K < 0 || D < 0 || N < 0 || R < 0 || H < 0 || W < 0) return VMB_ERR_INVALID_ARG;
    long long n = 0, nbc = 0;
    if (!count(&n, {B, K, D, H, W}) || !count(&nbc, {B, K, N > 0 ? N : 1, H, W})) return VMB_ERR_INVALID_ARG;
    if (n == 0) return VMB_OK;
    if ((long long)H * W > INT_MAX) return VMB_ERR_UNSUPPORTED;
    if (N < 1 || R < 1) return VMB_ERR_INVALID_ARG;
    if (N > 16 || R > 16) return VMB_ERR_UNSUPPORTED;
    long long rows = 0;
    if (!count(&rows, {B, K, D}) || rows > INT_MAX / 2) return VMB_ERR_UNSUPPORTED;
    if (!u || !WB || !WC || !Wz || !Wup || !Bs || !Cs || !delta_raw) return VMB_ERR_INVALID_ARG;
    const size_t es = esize(dtype);
    if (!aligned(u, es) || !aligned(Bs, es) || !aligned(Cs, es) || !aligned(delta_raw, es) || !aligned(WB, 4) ||
        !aligned(WC, 4) || !aligned(Wz, 4) || !aligned(Wup, 4))
        return VMB_ERR_MISALIGNED;
    SelArgs a{u, WB, WC, Wz, Wup, Bs, Cs, delta_raw, B, K, D, N, R, H * W, dtype};
    return launch_selection(a, stream);
}

vmb_status vmb_selection_lowrank_fwd(const void* u, const float* WB, const float* WC, const float* Wz, void* Bs,
                                     void* Cs, float* z, int B, int K, int D, int N, int R, int H, int W,
                                     vmb_dtype dtype, cudaStream_t stream) {
    if (!dtype_ok(dtype) || B < 0 || K < 0 || D < 0 || N < 0 || R < 0 || H < 0 || W < 0) return VMB_ERR_INVALID_ARG;
    long long n = 0, nbc = 0;
    if (!count(&n, {B, K, D, H, W}) || !count(&nbc, {B, K, N > 0 ? N : 1, H, W})) return VMB_ERR_INVALID_ARG;
    if (n == 0) return VMB_OK;
    if ((long long)H * W > INT_MAX) return VMB_ERR_UNSUPPORTED;
    if (N < 1 || R < 1) return VMB_ERR_INVALID_ARG;
    if (N > 16 || R > 16) return VMB_ERR_UNSUPPORTED;
    long long rows = 0;
    if (!count(&rows, {B, K, D}) || rows > INT_MAX / 2) return VMB_ERR_UNSUPPORTED;
    if (!u || !WB || !WC || !Wz || !Bs || !Cs || !z) return VMB_ERR_INVALID_ARG;
    const size_t es = esize(dtype);
    if (!aligned(u, es) || !aligned(Bs, es) || !aligned(Cs, es) || !aligned(z, 4) || !aligned(WB, 4) ||
        !aligned(WC, 4) || !aligned(Wz, 4))
        return VMB_ERR_MISALIGNED;
    SelArgs a{u, WB, WC, Wz, nullptr, Bs, Cs, nullptr, B, K, D, N, R, H * W, dtype};
    a.z = z;
    return launch_selection(a, stream);
}

size_t vmb_mean_scan_bwd_workspace_bytes(int B, int K, int D, int N, int H, int W, int groups, vmb_dtype dtype) {
    if (H < 0 || W < 0 || (long long)H * W > INT_MAX) return 0;
    static const float dummy[4] = {0, 0, 0, 0};
    float* dm = const_cast<float*>(dummy);
    MeanBwdArgs a{dummy, dummy, dummy, dummy, dummy, dummy, dummy, dummy, nullptr, dm, dm, dm, dm, dm, dm, dm,
                  B, K, D, N, H * W, groups, VMB_FLAG_SOFTPLUS, dtype, nullptr, 0};
    bool empty = false;
    if (check_bwd(a, &empty) != VMB_OK) return 0;
    if (empty) return 256;
    return mean_bwd_workspace_bytes(B, K, D, N, (long long)H * W, groups);
}

vmb_status vmb_mean_scan_bwd(const void* u, const void* delta, const float* A, const void* Bs, const void* Cs,
                             const float* Dskip, const float* delta_bias, const void* gy, const float* saved,
                             void* gu, void* gdelta,
                             float* gA, void* gBs, void* gCs, float* gDskip, float* gdelta_bias, int B, int K, int D,
                             int N, int H, int W, int groups, unsigned flags, vmb_dtype dtype, void* workspace,
                             size_t workspace_bytes, cudaStream_t stream) {
    if (H < 0 || W < 0) return VMB_ERR_INVALID_ARG;
    if ((long long)H * W > INT_MAX) return VMB_ERR_UNSUPPORTED;
    MeanBwdArgs a{u, delta, A, Bs, Cs, Dskip, delta_bias, gy, saved, gu, gdelta, gA, gBs, gCs, gDskip, gdelta_bias,
                  B, K, D, N, H * W, groups, flags, dtype, workspace, workspace_bytes};
    bool empty = false;
    vmb_status s = check_bwd(a, &empty);
    if (s != VMB_OK || empty) return s;
    if (!workspace) return VMB_ERR_WORKSPACE;
    if (!aligned(workspace, 256)) return VMB_ERR_MISALIGNED;
    if (workspace_bytes < mean_bwd_workspace_bytes(B, K, D, N, (long long)H * W, groups)) return VMB_ERR_WORKSPACE;
    return launch_mean_bwd(a, stream);
}

vmb_status vmb_read_status(void* workspace, cudaStream_t stream) {
    if (!workspace) return VMB_ERR_INVALID_ARG;
    if (!aligned(workspace, 256)) return VMB_ERR_MISALIGNED;
    WsHeader* hdr = static_cast<WsHeader*>(workspace);
    unsigned err = 0;
    if (cudaMemcpyAsync(&err, &hdr->err, sizeof(err), cudaMemcpyDeviceToHost, stream) != cudaSuccess)
        return VMB_ERR_CUDA;
    if (cudaStreamSynchronize(stream) != cudaSuccess) return VMB_ERR_CUDA;
    if (err == 0) return VMB_OK;
    if (cudaMemsetAsync(&hdr->err, 0, sizeof(unsigned), stream) != cudaSuccess) return VMB_ERR_CUDA;
    if (cudaStreamSynchronize(stream) != cudaSuccess) return VMB_ERR_CUDA;
    return (err & kErrTimeout) ? VMB_ERR_TIMEOUT : VMB_ERR_BOUNDS;
}

const char* vmb_status_string(vmb_status s) {
    switch (s) {
    case VMB_OK: return "ok";
    case VMB_ERR_INVALID_ARG: return "invalid argument";
    case VMB_ERR_MISALIGNED: return "misaligned pointer";
    case VMB_ERR_UNSUPPORTED: return "unsupported problem";
    case VMB_ERR_WORKSPACE: return "workspace missing or too small";
    case VMB_ERR_CUDA: return "CUDA error";
    case VMB_ERR_TIMEOUT: return "device wait timed out";
    case VMB_ERR_BOUNDS: return "device bounds check failed";
    }
    return "unknown status";
}

int vmb_version(void) { return 100; }

int vmb_testing_force_full_plan(int shape, int chunks) {
    g_force_chunks.store(chunks, std::memory_order_relaxed);
    g_force_shape.store(shape < 0 ? -1 : shape, std::memory_order_relaxed);
    return 0;
}

int vmb_testing_force_mean_chunk(int tc) {
    if (tc != 0 && tc != 32 && tc != 64 && tc != 128) return 1;
    g_force_tc.store(tc, std::memory_order_relaxed);
    return 0;
}

}  // extern "C"
