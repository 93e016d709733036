// vmb_internal.h - host-side plumbing between the C ABI (vmb_abi.cu) and the
// kernel launchers (cross_scan_merge.cu, full_scan.cu, mean_scan.cu).
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "vmb.h"

namespace vmb {

// One scan problem as the ABI received it (shapes already validated).
struct ScanArgs {
    const void* u;
    const void* delta;
    const float* A;
    const void* Bs;
    const void* Cs;
    const float* Dskip;
    const float* bias;
    void* y;
    float* ybar;  // mean path only (may be null)
    int B, K, D, N, L;
    unsigned flags;
    vmb_dtype dtype;
    void* ws;
    size_t ws_bytes;
    bool no_bcast = false;  // mean path fused with the cross-merge: ybar only, no y
    int bc_group = 1;       // grouped basis: K and D above are K*G and D/G; B / C rows per G sequences
    int gather_h = 0;       // > 0: u is the map x [B, D, H, W] (H = gather_h, K = 4) and u_t its transpose
                            // [B, D, W, H]; directions 0 / 2 read x, 1 / 3 read u_t (no materialised
                            // cross-scan)
    const void* u_t = nullptr;
    float* saved = nullptr;  // mean path: the group means kept for the backward, [B*K][N + 1][L] fp32
    const float* Wup = nullptr;  // full path, low-rank Delta: delta is z [B*K][R][L] fp32 and
    int R = 0;                   // delta_raw = Wup z (Wup [K][D][R]); warp-specialised plans only
};

// Execution plan of an L-chunked scan: how the (sequence, chunk) grid is cut
// and how much workspace its look-back needs.  Deterministic for a given
// problem, build and device, so that the workspace query and the launch agree.
struct ScanPlan {
    int np;            // padded state count (1, 2, 4, 8, 16)
    int split;         // tile-shape index (full path)
    int tile_rows;     // channels per CTA (full path) or 0 (mean path)
    int tiles_per_bk;  // channel tiles per (b, k)   (full path)
    int n_seq;         // independent sequences: channel tiles (full) or (b, k) pairs (mean)
    int n_chunks;      // chunks along L per sequence
    int chunk_len;     // steps per chunk (a multiple of the stage length)
    size_t state_floats;  // floats of one chunk's published state (per array)
    size_t ws_bytes;      // total workspace bytes
    bool early = true;    // may be launched before the previous kernel of the stream completes
};

inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Workspace layout: [header 256 B][flags n_seq*n_chunks u32][agg_P][agg_H][inc_H]
struct WsLayout {
    size_t flags_off, aggP_off, aggH_off, incH_off, total;
};
inline WsLayout ws_layout(const ScanPlan& p) {
    WsLayout w;
    size_t slots = (size_t)p.n_seq * (size_t)p.n_chunks;
    w.flags_off = 256;
    w.aggP_off = align_up(w.flags_off + slots * 4, 256);
    size_t arr = align_up(slots * p.state_floats * 4, 256);
    w.aggH_off = w.aggP_off + arr;
    w.incH_off = w.aggH_off + arr;
    w.total = w.incH_off + arr;
    if (p.n_chunks <= 1) w.total = 256;  // single-chunk plans only use the header
    return w;
}

// The paper's scan-only setting (Sec. 4): discretisation into materialised
// fp32 operands, then the scan alone.
struct DiscArgs {
    const void* u;
    const void* delta;
    const float* A;
    const void* Bs;
    const float* bias;
    float* dA;   // [B][K][D][N][L], or [B][K][N][L] for the channel means
    float* dBu;  // same shape as dA
    int B, K, D, N, L;
    unsigned flags;
    vmb_dtype dtype;
};
struct OnlyArgs {
    const float* dA;   // [B][K][Dm][N][L]
    const float* dBu;  // [B][K][Dm][N][L]
    const void* Cs;    // [B][K][N][L], dtype
    float* y;          // [B][K][Dm][L]
    int B, K, Dm, N, L;
    vmb_dtype dtype;
};

// The selection functions of Eq. 6 (B, C and the raw Delta from the input).
struct SelArgs {
    const void* u;     // [B][K][D][L], dtype
    const float* WB;   // [K][N][D]
    const float* WC;   // [K][N][D]
    const float* Wz;   // [K][R][D]
    const float* Wup;  // [K][D][R]
    void* Bs;          // [B][K][N][L], dtype
    void* Cs;          // [B][K][N][L], dtype
    void* delta_raw;   // [B][K][D][L], dtype
    int B, K, D, N, R, L;
    vmb_dtype dtype;
    float* z = nullptr;  // not null: z [B][K][R][L] fp32 written instead of delta_raw (Wup unused)
};

// Gradients of the (grouped) channel-mean scan.
struct MeanBwdArgs {
    const void* u;
    const void* delta;  // raw Delta (before bias and softplus)
    const float* A;
    const void* Bs;
    const void* Cs;
    const float* Dskip;
    const float* bias;
    const void* gy;
    const float* saved;  // the forward's group means, or null (recomputed)
    void* gu;
    void* gdelta;
    float* gA;
    void* gBs;
    void* gCs;
    float* gDskip;
    float* gbias;
    int B, K, D, N, L, groups;
    unsigned flags;
    vmb_dtype dtype;
    void* ws;
    size_t ws_bytes;
};

int device_sm_count();

// The argument checks of the scan entry points (shapes, flags, pointers,
// alignment); *empty is set for a problem with no elements.
vmb_status validate_scan(const ScanArgs& a, bool mean, bool* empty);

// Test-only plan overrides (vmb_testing.h); -1 / 0 when unset.
int forced_full_shape(int* chunks);
int forced_mean_chunk();

vmb_status plan_full(const ScanArgs& a, ScanPlan* plan);
vmb_status plan_mean(const ScanArgs& a, ScanPlan* plan);
vmb_status launch_full(const ScanArgs& a, const ScanPlan& plan, cudaStream_t stream);
int full_plan_launches(const ScanPlan& plan);  // kernels launch_full starts for this plan
// Whether launch_full can read the plan's u gathered from the map (ScanArgs::gather_h)
// or expand a low-rank Delta (ScanArgs::R): the warp-specialised plans.
bool full_plan_gathers(const ScanPlan& plan);
// out [B,K,D,L] (dtype) = Wup z, the raw Deltas of the low-rank form.
vmb_status launch_lowrank_expand(const float* z, const float* Wup, void* out, int B, int K, int D, int R, int L,
                                 vmb_dtype dt, cudaStream_t stream);
vmb_status launch_mean(const ScanArgs& a, const ScanPlan& plan, cudaStream_t stream);
vmb_status launch_cross_scan(const void* x, void* xs, int B, int D, int H, int W, vmb_dtype dt,
                             cudaStream_t stream);
vmb_status launch_cross_merge(const void* ys, void* out, int B, int D, int H, int W, vmb_dtype dt,
                              cudaStream_t stream);
vmb_status launch_map_transpose(const void* x, void* xt, int B, int D, int H, int W, vmb_dtype dt,
                                cudaStream_t stream);
vmb_status launch_discretise(const DiscArgs& a, bool mean, cudaStream_t stream);
vmb_status launch_selection(const SelArgs& a, cudaStream_t stream);
size_t mean_bwd_workspace_bytes(long long B, long long K, long long D, long long N, long long L, long long G);
vmb_status launch_mean_bwd(const MeanBwdArgs& a, cudaStream_t stream);
vmb_status launch_scan_only(const OnlyArgs& a, cudaStream_t stream);
vmb_status launch_mean_merge(const void* x, const float* ybar, const float* Dskip, void* out, int B, int D, int H,
                             int W, bool per_channel_skip, vmb_dtype dt, cudaStream_t stream);

}  // namespace vmb
