// mean_backward.cu - gradients of the (grouped) channel-mean scan for sm_103a.
//
// The reverse-mode derivative of Eq. 9's forward (the VMeanba scan, Sec. 2.2;
// with G > 1 channel groups the grouped basis of Sec. 2.1 / Eq. 8), Euler
// Bbar and the per-channel skip term.  Per sequence s = (b, k, g) of M = D / G
// channels d (parameter index c = k D + d):
//   delta_d = softplus(raw_d + bias_c), Abar_n = (1/M) sum_d exp(delta_d A_cn),
//   sm = (1/M) sum_d delta_d u_d, h_n(t) = Abar_n(t) h_n(t-1) + B_n(t) sm(t),
//   y_d = sum_n C_n h_n + Dskip_c u_d.
// Given gy = dLoss/dy, with lam_n(t) = dLoss/dh_n(t) run backward in time,
//   lam_n(t) = C_n(t) gyb(t) + Abar_n(t+1) lam_n(t+1),   gyb(t) = sum_d gy_d(t),
//   gC_n(t) += gyb(t) h_n(t), gB_n(t) += lam_n(t) sm(t),
//   gAbar_n(t) = lam_n(t) h_n(t-1), gs(t) = sum_n lam_n(t) B_n(t),
// and per channel
//   gu_d = Dskip_c gy_d + gs delta_d / M,
//   graw_d = softplus'(raw_d + bias_c) (gs u_d + sum_n gAbar_n A_cn exp(delta_d A_cn)) / M,
//   gA_cn += gAbar_n delta_d exp(delta_d A_cn) / M, gDskip_c += gy_d u_d, gbias_c += graw_d.
//
// Both recurrences are linear, so they are scanned in chunks of kLC steps:
// with nu_n(t) = Abar_n(t) lam_n(t) the adjoint becomes
//   nu_n(t) = Abar_n(t) nu_n(t+1) + Abar_n(t) C_n(t) gyb(t),
// the same form as the forward one run the other way, and a chunk is summed up
// by the product P of its Abar, the forward state it reaches from zero and the
// adjoint it reaches from zero.  Six launches, every reduction in a fixed
// order (results are deterministic):
//   1. per (sequence, kRT steps): the group means Abar, sm and the summed
//      output gradient gyb (a thread per step, the group's channels split in
//      two, their A rows staged in shared memory);
//   2. per (sequence, chunk): the chunk summaries (a warp per chunk: lanes 0-15
//      the forward states, lanes 16-31 the adjoint);
//   3. per (sequence, state): the carries into every chunk, folded in chunk order;
//   4. per (sequence, chunk): both recurrences again from their carries into
//      shared memory, then gAbar / M, gs / M, gB and gC written coalesced;
//   5. per (channel, span of steps): the chain rule through the mean and the
//      softplus, gu and graw, and partial sums of gA, gDskip and gbias per
//      (batch, span);
//   6. the partial sums added in (batch, span) order (and gB, gC over the groups).
#include "vmb_common.cuh"
#include "vmb_internal.h"

namespace vmb {
namespace {

constexpr int kNP = 16;           // states per sequence as stored (N <= 16, zero padded)
constexpr int kRT = 128;          // steps per CTA of launch 1
constexpr int kRThreads = 2 * kRT;
constexpr int kCG = 256;          // channels whose A rows are staged at a time (launch 1)
constexpr int kPF = 4;            // channels a launch-1 thread has in flight
constexpr int kLC = 32;           // steps per scan chunk (launches 2-4)
constexpr int kSWarps = 8;        // chunks per CTA of launches 2 and 4
constexpr int kSB = 16;           // steps whose loads a launch-2/4 lane issues together
constexpr int kCThreads = 128;    // threads per CTA of launch 5
constexpr int kSlots = 4;         // launch-5 threads per channel
constexpr int kCCh = kCThreads / kSlots;  // channels per CTA of launch 5
constexpr int kCV = 2 * kSlots;   // steps per group of launch 5 (two per slot)
constexpr int kTS = 16;           // steps per shared-memory stage of launch 5
constexpr int kNS = 4;            // stages of launch 5
constexpr int kRowE = 24;         // staged input row stride (elements)
constexpr int kGabE = 20;         // staged gAbar row stride (floats)
constexpr int kSpanTarget = 4096; // launch-5 CTAs aimed for when splitting the steps
constexpr int kMinSpan = 256;     // fewest steps per launch-5 span
constexpr float kLn2 = 0.6931471805599453f;

struct BwdParams {
    const void* u;
    const void* raw;
    const float* A;
    const void* Bs;
    const void* Cs;
    const float* Dskip;
    const float* bias;
    const void* gy;
    void* gu;
    void* graw;
    float* gA;
    void* gB;
    void* gC;
    float* gDskip;
    float* gbias;
    int B, K, D, N, L, G, M;  // M = D / G channels per sequence
    int softplus_on;
    int nch;                  // scan chunks per sequence
    int nspan, span_len;      // launch-5 spans of the steps
    int vec;                  // rows of Abar, sm, gyb, B, C allow 4-step vector loads
    bool saved;               // ms holds the forward's means: launch 1 sums gy only
    // workspace arrays (fp32)
    float* ms;    // [S][N + 1][L]: Abar_n rows, then sm (the forward's saved means, or launch 1's)
    float* gyb;   // [S][L]
    float* sumP;  // [S][nch][kNP] product of the chunk's Abar
    float* sumH;  // [S][nch][kNP] forward state from zero; after launch 3 the state entering the chunk
    float* sumV;  // [S][nch][kNP] adjoint nu from zero; after launch 3 nu just past the chunk
    float* gab;   // [S][L][kNP] gAbar / M
    float* gs;    // [S][L] gs / M
    float* gBw;   // [S][kNP][L] (groups > 1): per-group contributions to gB
    float* gCw;   // [S][kNP][L]
    float* pA;    // [B][nspan][K D][kNP] partial sums
    float* pD;    // [B][nspan][K D]
    float* pb;    // [B][nspan][K D]
};

// Launch-5 spans: enough (batch, channel block, span) CTAs to fill the GPU a
// few times over, every span a multiple of kTS steps and at least kMinSpan.
void bwd_spans(long long B, long long K, long long D, long long L, long long G, int* nspan, int* span_len) {
    const long long ctas = B * K * G * ((D / G + kCCh - 1) / kCCh);
    long long want = ctas > 0 ? (kSpanTarget + ctas - 1) / ctas : 1;
    const long long most = L / kMinSpan > 1 ? L / kMinSpan : 1;
    if (want > most) want = most;
    if (want < 1) want = 1;
    long long len = (L + want - 1) / want;
    len = (len + kTS - 1) / kTS * kTS;
    *span_len = (int)len;
    *nspan = (int)((L + len - 1) / len);
}

// Workspace layout (256-byte aligned arrays).
struct BwdLayout {
    size_t ms, gyb, sumP, sumH, sumV, gab, gs, gBw, gCw, pA, pD, pb, total;
    int nch, nspan, span_len;
};
BwdLayout bwd_layout(long long B, long long K, long long D, long long N, long long L, long long G) {
    const long long S = B * K * G;
    BwdLayout w{};
    w.nch = (int)((L + kLC - 1) / kLC);
    bwd_spans(B, K, D, L, G, &w.nspan, &w.span_len);
    size_t o = 0;
    auto take = [&](size_t bytes) {
        const size_t at = o;
        o = align_up(o + bytes, 256);
        return at;
    };
    w.ms = take((size_t)S * (N + 1) * L * 4);
    w.gyb = take((size_t)S * L * 4);
    w.sumP = take((size_t)S * w.nch * kNP * 4);
    w.sumH = take((size_t)S * w.nch * kNP * 4);
    w.sumV = take((size_t)S * w.nch * kNP * 4);
    w.gab = take((size_t)S * L * kNP * 4);
    w.gs = take((size_t)S * L * 4);
    w.gBw = take(G > 1 ? (size_t)S * kNP * L * 4 : 0);
    w.gCw = take(G > 1 ? (size_t)S * kNP * L * 4 : 0);
    w.pA = take((size_t)B * w.nspan * K * D * kNP * 4);
    w.pD = take((size_t)B * w.nspan * K * D * 4);
    w.pb = take((size_t)B * w.nspan * K * D * 4);
    w.total = o;
    return w;
}

__device__ __forceinline__ float delta_of(float v, int softplus_on) { return softplus_on ? softplus(v) : v; }

// softplus'(v) = the logistic function 1 / (1 + e^-v), from e^-|v| (no overflow)
__device__ __forceinline__ float softplus_grad(float v) {
    const float e = ex2(-fabsf(v) * kLog2e);
    const float r = rcp(1.0f + e);
    return v >= 0.0f ? r : e * r;
}

// ---------------------------------------------------------------- launch 1
// CTA = one sequence x kRT steps; thread (t, half) reduces every other channel
// of the group at step t, kPF channels in flight; the two halves are added in
// shared memory and written as [n][t] rows.
template <typename T>
__global__ void __launch_bounds__(kRThreads, 3) bwd_reduce_kernel(const BwdParams p) {
    __shared__ __align__(16) float s_a2[kCG * kNP];  // A log2 e of kCG channels
    __shared__ float s_bias[kCG];
    __shared__ float red[2][kNP + 2][kRT];
    pdl_wait();
    pdl_launch_dependents();
    const int L = p.L, N = p.N, M = p.M;
    const int nlb = (L + kRT - 1) / kRT;
    const int seq = blockIdx.x / nlb;  // (b, k, g)
    const int t0 = (blockIdx.x % nlb) * kRT;
    const int rt = threadIdx.x % kRT, half = threadIdx.x / kRT;
    const int t = t0 + rt;
    const bool tv = t < L;
    const int bk = seq / p.G, g = seq % p.G, k = bk % p.K;
    const size_t row0 = (size_t)bk * p.D + (size_t)g * M;  // first (b, k, d) row of the group
    const size_t col = row0 * L + (tv ? t : 0);
    const T* raw = static_cast<const T*>(p.raw) + col;
    const T* u = static_cast<const T*>(p.u) + col;
    const T* gy = static_cast<const T*>(p.gy) + col;
    const uint64_t stream = l2_evict_first();
    float2 acc[kNP / 2];  // states as pairs (n, n + 1) for the packed f32x2 operations
#pragma unroll
    for (int m = 0; m < kNP / 2; ++m) acc[m] = make_float2(0.0f, 0.0f);
    float su = 0.0f, sg = 0.0f;
    const int c0 = k * p.D + g * M;
    const int cs = 2 * L;  // between a thread's consecutive channels
    for (int j0 = 0; j0 < M; j0 += kCG) {
        const int gn = min(kCG, M - j0);
        if (j0 > 0) __syncthreads();  // the previous tables are no longer read
        const float* Ag = p.A + (size_t)(c0 + j0) * N;
        for (int i = threadIdx.x; i < kCG * kNP; i += kRThreads) {
            const int r = i / kNP, n = i % kNP;
            s_a2[i] = (r < gn && n < N) ? __ldg(Ag + (size_t)r * N + n) * kLog2e : 0.0f;
        }
        for (int i = threadIdx.x; i < kCG; i += kRThreads) s_bias[i] = i < gn ? __ldg(p.bias + c0 + j0 + i) : 0.0f;
        __syncthreads();
        if (!tv) continue;
        // this thread's channels of the group: j = j0 + half + 2 i, i < nj
        const int nj = (gn - half + 1) / 2;
        // offsets within the group are 32-bit (D L < 2^31, checked by the host)
        const int first = (j0 + half) * L;
        const T* rb = raw + first;
        const T* ub = u + first;
        const T* gb = gy + first;
        float vr[kPF], vu[kPF], vg[kPF];
        auto load = [&](int i0, float (&r)[kPF], float (&uu)[kPF], float (&gg)[kPF]) {
            const int o0 = i0 * cs;
            if (i0 + kPF <= nj) {  // the whole batch is in range: no per-channel checks
#pragma unroll
                for (int q = 0; q < kPF; ++q) {
                    const int o = o0 + q * cs;
                    r[q] = ld_hint(rb + o, stream);
                    uu[q] = ld_hint(ub + o, stream);
                    gg[q] = ld_hint(gb + o, stream);
                }
            } else {
#pragma unroll
                for (int q = 0; q < kPF; ++q) {
                    const bool ok = i0 + q < nj;
                    const int o = o0 + q * cs;
                    r[q] = ok ? ld_hint(rb + o, stream) : 0.0f;
                    uu[q] = ok ? ld_hint(ub + o, stream) : 0.0f;
                    gg[q] = ok ? ld_hint(gb + o, stream) : 0.0f;
                }
            }
        };
        auto reduce_one = [&](float vrq, float vuq, float vgq, int jj) {
            const float dl = delta_of(vrq + s_bias[jj], p.softplus_on);
            const float2 dl2 = make_float2(dl, dl);
            const float* a2 = s_a2 + jj * kNP;  // broadcast reads: every lane has the same channel
#pragma unroll
            for (int n = 0; n < kNP; n += 4) {
                const float4 qa = *reinterpret_cast<const float4*>(a2 + n);
                const float2 e01 = __fmul2_rn(dl2, make_float2(qa.x, qa.y));
                const float2 e23 = __fmul2_rn(dl2, make_float2(qa.z, qa.w));
                acc[n / 2] = __fadd2_rn(acc[n / 2], make_float2(ex2(e01.x), ex2(e01.y)));
                acc[n / 2 + 1] = __fadd2_rn(acc[n / 2 + 1], make_float2(ex2(e23.x), ex2(e23.y)));
            }
            su = fmaf(dl, vuq, su);
            sg += vgq;
        };
        load(0, vr, vu, vg);
        for (int i0 = 0; i0 < nj; i0 += kPF) {
            float nr[kPF], nu[kPF], ng[kPF];
            load(i0 + kPF, nr, nu, ng);
            if (i0 + kPF <= nj) {
#pragma unroll
                for (int q = 0; q < kPF; ++q) reduce_one(vr[q], vu[q], vg[q], half + 2 * (i0 + q));
            } else {
#pragma unroll
                for (int q = 0; q < kPF; ++q)
                    if (i0 + q < nj) reduce_one(vr[q], vu[q], vg[q], half + 2 * (i0 + q));
            }
#pragma unroll
            for (int q = 0; q < kPF; ++q) {
                vr[q] = nr[q];
                vu[q] = nu[q];
                vg[q] = ng[q];
            }
        }
    }
#pragma unroll
    for (int m = 0; m < kNP / 2; ++m) {
        red[half][2 * m][rt] = acc[m].x;
        red[half][2 * m + 1][rt] = acc[m].y;
    }
    red[half][kNP][rt] = su;
    red[half][kNP + 1][rt] = sg;
    __syncthreads();
    const float inv = 1.0f / (float)M;
    for (int i = threadIdx.x; i < (kNP + 2) * kRT; i += kRThreads) {
        const int r = i / kRT, tt = i % kRT;
        if (t0 + tt >= L) continue;
        if (r >= N && r < kNP) continue;  // padding states
        const float v = red[0][r][tt] + red[1][r][tt];
        if (r < kNP)
            p.ms[((size_t)seq * (N + 1) + r) * L + t0 + tt] = v * inv;
        else if (r == kNP)
            p.ms[((size_t)seq * (N + 1) + N) * L + t0 + tt] = v * inv;
        else
            p.gyb[(size_t)seq * L + t0 + tt] = v;
    }
}

// Launch 1 when the forward kept its means: only gyb = sum_d gy_d per step
// (CTA = one sequence x kRT steps, the group's channels split in two halves,
// kPF2 channels in flight per thread).
constexpr int kPF2 = 8;
template <typename T>
__global__ void __launch_bounds__(kRThreads) bwd_gysum_kernel(const BwdParams p) {
    __shared__ float red[2][kRT];
    pdl_wait();
    pdl_launch_dependents();
    const int L = p.L, M = p.M;
    const int nlb = (L + kRT - 1) / kRT;
    const int seq = blockIdx.x / nlb;
    const int t0 = (blockIdx.x % nlb) * kRT;
    const int rt = threadIdx.x % kRT, half = threadIdx.x / kRT;
    const int t = t0 + rt;
    const bool tv = t < L;
    const int bk = seq / p.G, g = seq % p.G;
    const T* gy = static_cast<const T*>(p.gy) + ((size_t)bk * p.D + (size_t)g * M + half) * L + (tv ? t : 0);
    const uint64_t stream = l2_evict_first();
    const int nj = (M - half + 1) / 2;  // channels half + 2 i, i < nj
    const int cs = 2 * L;
    float s = 0.0f;
    if (tv) {
        int i0 = 0;
        for (; i0 + kPF2 <= nj; i0 += kPF2) {
            float v[kPF2];
#pragma unroll
            for (int q = 0; q < kPF2; ++q) v[q] = ld_hint(gy + (i0 + q) * cs, stream);
#pragma unroll
            for (int q = 0; q < kPF2; ++q) s += v[q];
        }
        for (; i0 < nj; ++i0) s += ld_hint(gy + i0 * cs, stream);
    }
    red[half][rt] = s;
    __syncthreads();
    if (half == 0 && tv) p.gyb[(size_t)seq * L + t] = red[0][rt] + red[1][rt];
}

// One step of either chunk recurrence, in a form both halves of a warp run:
// the forward state h = a h + pq (stored: h), the adjoint nu = a (nu + pq)
// (stored: lam = nu + pq).  Returns the stored value; x becomes the new carry.
__device__ __forceinline__ float chunk_step(int dir, float a, float pq, float& x) {
    const float r = dir ? x + pq : fmaf(a, x, pq);
    x = dir ? a * r : r;
    return r;
}

// Four consecutive elements of a row as fp32 (16 bytes fp32, 8 bytes bf16);
// the caller guarantees the alignment.
__device__ __forceinline__ float4 ld4v(const float* q) { return *reinterpret_cast<const float4*>(q); }
__device__ __forceinline__ float4 ld4v(const __nv_bfloat16* q) {
    const uint2 w = *reinterpret_cast<const uint2*>(q);
    return make_float4(__uint_as_float(w.x << 16), __uint_as_float(w.x & 0xffff0000u), __uint_as_float(w.y << 16),
                       __uint_as_float(w.y & 0xffff0000u));
}

// Steps ts .. ts + kSB - 1 of a lane's rows, all loads issued before any is
// used: Abar_n(t) and the input term (B_n sm forward, C_n gyb adjoint).  Steps
// at or past tend, and padding states (n >= N), give the identity step
// (a = 1, term 0) and read no Abar.
// With vec (rows 4-element aligned, ts a multiple of 4) whole quads are read
// as vectors.  rev: the adjoint lanes get the batch in reverse step order.
template <typename T>
__device__ __forceinline__ void batch_load(const float* ab, const T* pr, const float* qr, bool nv, bool vec, bool rev,
                                           int ts, int tend, float (&a)[kSB], float (&pq)[kSB]) {
    float pv[kSB], qv[kSB];
#pragma unroll
    for (int q = 0; q < kSB / 4; ++q) {
        const int t = ts + 4 * q;
        if (vec && t + 4 <= tend) {
            const float4 av = nv ? ld4v(ab + t) : make_float4(1.0f, 1.0f, 1.0f, 1.0f), qq = ld4v(qr + t);
            const float4 pp = nv ? ld4v(pr + t) : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            a[4 * q] = av.x, a[4 * q + 1] = av.y, a[4 * q + 2] = av.z, a[4 * q + 3] = av.w;
            qv[4 * q] = qq.x, qv[4 * q + 1] = qq.y, qv[4 * q + 2] = qq.z, qv[4 * q + 3] = qq.w;
            pv[4 * q] = pp.x, pv[4 * q + 1] = pp.y, pv[4 * q + 2] = pp.z, pv[4 * q + 3] = pp.w;
        } else {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const bool ok = t + i < tend;
                a[4 * q + i] = (ok && nv) ? ab[t + i] : 1.0f;
                pv[4 * q + i] = (ok && nv) ? io<T>::ld(pr + t + i) : 0.0f;
                qv[4 * q + i] = ok ? qr[t + i] : 0.0f;
            }
        }
    }
#pragma unroll
    for (int i = 0; i < kSB; ++i) pq[i] = pv[i] * qv[i];
    // the two halves of a warp differ in rev: selects, not a branch
#pragma unroll
    for (int i = 0; i < kSB / 2; ++i) {
        const float x = a[i], y = pq[i], xr = a[kSB - 1 - i], yr = pq[kSB - 1 - i];
        a[i] = rev ? xr : x, pq[i] = rev ? yr : y;
        a[kSB - 1 - i] = rev ? x : xr, pq[kSB - 1 - i] = rev ? y : yr;
    }
}

// ---------------------------------------------------------------- launch 2
// A warp per (sequence, chunk): lane n < 16 runs the forward states from zero
// (and the product of the chunk's Abar), lane 16 + n the adjoint from zero.
template <typename T>
__global__ void __launch_bounds__(32 * kSWarps) bwd_summary_kernel(const BwdParams p, int n_pairs) {
    pdl_wait();
    pdl_launch_dependents();
    const int pair = blockIdx.x * kSWarps + threadIdx.x / 32;
    if (pair >= n_pairs) return;  // the whole warp: nothing below synchronises the block
    const int lane = threadIdx.x % 32, dir = lane / 16, n = lane % 16;
    const int L = p.L, N = p.N;
    const int seq = pair / p.nch, ch = pair % p.nch;
    const int t0 = ch * kLC, len = min(kLC, L - t0);
    const bool nv = n < N;
    const float* ab = p.ms + ((size_t)seq * (N + 1) + (nv ? n : 0)) * L;
    const T* pr = static_cast<const T*>(dir ? p.Cs : p.Bs) + ((size_t)(seq / p.G) * N + (nv ? n : 0)) * L;
    const float* qr = dir ? p.gyb + (size_t)seq * L : p.ms + ((size_t)seq * (N + 1) + N) * L;
    // forward lanes take the chunk's batches in order, adjoint lanes in reverse
    const int nb = (len + kSB - 1) / kSB;
    float x = 0.0f, P = 1.0f;
    for (int bi = 0; bi < nb; ++bi) {
        float a[kSB], pq[kSB];
        batch_load<T>(ab, pr, qr, nv, p.vec, dir, t0 + kSB * (dir ? nb - 1 - bi : bi), t0 + len, a, pq);
#pragma unroll
        for (int i = 0; i < kSB; ++i) {
            chunk_step(dir, a[i], pq[i], x);
            P *= a[i];
        }
    }
    const size_t idx = (size_t)pair * kNP + n;
    if (dir == 0) {
        p.sumP[idx] = P;
        p.sumH[idx] = x;
    } else {
        p.sumV[idx] = x;
    }
}

// ---------------------------------------------------------------- launch 3
// A thread per (sequence, direction, state): the chunk summaries folded in
// chunk order (forward) or reverse chunk order (adjoint), each replaced by the
// carry that enters its chunk.
__global__ void __launch_bounds__(256) bwd_carry_kernel(const BwdParams p, int n_lanes) {
    pdl_wait();
    pdl_launch_dependents();
    const int i = blockIdx.x * 256 + threadIdx.x;
    if (i >= n_lanes) return;
    const int seq = i / 32, dir = (i / 16) % 2, n = i % 16;
    const size_t base = (size_t)seq * p.nch * kNP + n;
    // forward: chunks in order, sumH becomes h(t0 - 1); adjoint: chunks in
    // reverse, sumV becomes nu(t1), t1 the first step after the chunk.  kSB
    // chunks' summaries are loaded before any is replaced.
    float* sv = dir ? p.sumV : p.sumH;
    float x = 0.0f;
    for (int j0 = 0; j0 < p.nch; j0 += kSB) {
        float hv[kSB], pv[kSB];
#pragma unroll
        for (int j = 0; j < kSB; ++j) {
            const int ch = dir ? p.nch - 1 - (j0 + j) : j0 + j;
            const bool ok = j0 + j < p.nch;
            hv[j] = ok ? sv[base + (size_t)ch * kNP] : 0.0f;
            pv[j] = ok ? p.sumP[base + (size_t)ch * kNP] : 0.0f;
        }
#pragma unroll
        for (int j = 0; j < kSB; ++j) {
            if (j0 + j < p.nch) {
                const int ch = dir ? p.nch - 1 - (j0 + j) : j0 + j;
                sv[base + (size_t)ch * kNP] = x;
                x = fmaf(pv[j], x, hv[j]);
            }
        }
    }
}

// ---------------------------------------------------------------- launch 4
// A warp per (sequence, chunk): both recurrences again from their carries,
// h and lam kept in shared memory, then the per-step gradients written by the
// whole warp along the steps.
template <typename T>
__global__ void __launch_bounds__(32 * kSWarps) bwd_chunk_kernel(const BwdParams p, int n_pairs) {
    __shared__ float s_h[kSWarps][kLC + 1][kNP + 1];  // row i: h(t0 - 1 + i)
    __shared__ float s_l[kSWarps][kLC][kNP + 1];      // row i: lam(t0 + i)
    pdl_wait();
    pdl_launch_dependents();
    const int w = threadIdx.x / 32;
    const int pair = blockIdx.x * kSWarps + w;
    if (pair >= n_pairs) return;  // the whole warp: only warp-level barriers below
    const int lane = threadIdx.x % 32, dir = lane / 16, n = lane % 16;
    const int L = p.L, N = p.N;
    const int seq = pair / p.nch, ch = pair % p.nch;
    const int bk = seq / p.G;
    const int t0 = ch * kLC, len = min(kLC, L - t0);
    const bool nv = n < N;
    float(*hs)[kNP + 1] = s_h[w];
    float(*ls)[kNP + 1] = s_l[w];
    {
        const float* ab = p.ms + ((size_t)seq * (N + 1) + (nv ? n : 0)) * L;
        const T* pr = static_cast<const T*>(dir ? p.Cs : p.Bs) + ((size_t)bk * N + (nv ? n : 0)) * L;
        const float* qr = dir ? p.gyb + (size_t)seq * L : p.ms + ((size_t)seq * (N + 1) + N) * L;
        const size_t idx = (size_t)pair * kNP + n;
        float x = dir ? p.sumV[idx] : p.sumH[idx];
        if (dir == 0) hs[0][n] = x;
        const int nb = (len + kSB - 1) / kSB;
        // the row a lane stores step i of a batch in: forward h(t) at hs row
        // b0 + i + 1, adjoint lam(t) at ls row b0 + kSB - 1 - i (one store, no branch)
        const int rstep = dir ? -(kNP + 1) : kNP + 1;
        for (int bi = 0; bi < nb; ++bi) {
            const int b0 = kSB * (dir ? nb - 1 - bi : bi);  // first step of the batch within the chunk
            float a[kSB], pq[kSB];
            batch_load<T>(ab, pr, qr, nv, p.vec, dir, t0 + b0, t0 + len, a, pq);
            float* rowp = dir ? &ls[b0 + kSB - 1][n] : &hs[b0 + 1][n];
#pragma unroll
            for (int i = 0; i < kSB; ++i) {
                // steps past the chunk are identity steps; their rows (< kLC) are never read
                rowp[i * rstep] = chunk_step(dir, a[i], pq[i], x);
            }
        }
    }
    __syncwarp();
    const float invM = 1.0f / (float)p.M;
    // gAbar / M = lam h(t - 1) / M: the chunk's [t][n] rows are contiguous
    float* gab = p.gab + ((size_t)seq * L + t0) * kNP;
    for (int j = lane; j < len * kNP; j += 32) {
        const int i = j / kNP, m = j % kNP;
        gab[j] = m < N ? ls[i][m] * hs[i][m] * invM : 0.0f;
    }
    const T* Bb = static_cast<const T*>(p.Bs) + (size_t)bk * N * L;
    const float* smv = p.ms + ((size_t)seq * (N + 1) + N) * L;
    const float* gybv = p.gyb + (size_t)seq * L;
    for (int i = lane; i < len; i += 32) {
        const int t = t0 + i;
        float s = 0.0f;  // gs / M = sum_n lam_n B_n / M, in state order
        for (int m = 0; m < N; ++m) s = fmaf(ls[i][m], io<T>::ld(Bb + (size_t)m * L + t), s);
        p.gs[(size_t)seq * L + t] = s * invM;
    }
    // gC_n = gyb h_n, gB_n = lam_n sm: lanes along the steps of each [n][t] row
    constexpr int kPer = kLC / 32;  // steps per lane
    float gyl[kPer], sml[kPer];
#pragma unroll
    for (int r = 0; r < kPer; ++r) {
        const int i = lane + 32 * r;
        gyl[r] = i < len ? gybv[t0 + i] : 0.0f;
        sml[r] = i < len ? smv[t0 + i] : 0.0f;
    }
    for (int m = 0; m < N; ++m) {
#pragma unroll
        for (int r = 0; r < kPer; ++r) {
            const int i = lane + 32 * r;
            if (i >= len) continue;
            const int t = t0 + i;
            const float gc = gyl[r] * hs[i + 1][m], gb = ls[i][m] * sml[r];
            if (p.G == 1) {
                static_cast<T*>(p.gC)[((size_t)bk * N + m) * L + t] = io<T>::to(gc);
                static_cast<T*>(p.gB)[((size_t)bk * N + m) * L + t] = io<T>::to(gb);
            } else {
                p.gCw[((size_t)seq * kNP + m) * L + t] = gc;
                p.gBw[((size_t)seq * kNP + m) * L + t] = gb;
            }
        }
    }
}

// ---------------------------------------------------------------- launch 5
// Shared-memory stage of launch 5: kTS steps of the CTA's kCCh rows of raw,
// u and gy as stored (rows kRowE elements apart: the slots' 2-element reads
// of a warp hit distinct banks), gAbar / M rows kGabE floats apart and gs / M.
template <typename T>
struct ChanStage {
    static constexpr size_t in = (size_t)kCCh * kRowE * sizeof(T);  // one input array
    static constexpr size_t gab = 3 * in;
    static constexpr size_t gs = gab + (size_t)kTS * kGabE * 4;
    static constexpr size_t bytes = gs + (size_t)kTS * 4;
    static_assert(in % 16 == 0 && gs % 16 == 0 && bytes % 16 == 0, "16-byte aligned stage parts");
};

struct ChanRows {
    const void* in[3];  // raw, u, gy of the CTA's first channel (element offset of row 0)
    const float* gab;   // the group's gAbar / M, [L][kNP]
    const float* gs;    // the group's gs / M, [L]
    int nrows;          // valid channel rows of the CTA
    int L;
};

// Steps ts .. ts + kTS - 1 (zero past l1) into stage `st`: 16-byte async copies
// (VEC: rows, ts and l1 aligned to kCV, 16-byte aligned bases) or element loads.
template <typename T, bool VEC>
__device__ __forceinline__ void stage_chan(unsigned char* st, const ChanRows& r, int ts, int l1) {
    using CS = ChanStage<T>;
    float* sg = reinterpret_cast<float*>(st + CS::gab);
    float* ss = reinterpret_cast<float*>(st + CS::gs);
    if constexpr (VEC) {
        constexpr int EPC = 16 / (int)sizeof(T);  // elements per copy
        constexpr int CPR = kTS / EPC;            // copies per row
        for (int i = threadIdx.x; i < 3 * kCCh * CPR; i += kCThreads) {
            const int arr = i / (kCCh * CPR), row = (i / CPR) % kCCh, q = i % CPR;
            const int t = ts + q * EPC;
            const bool ok = row < r.nrows && t < l1;
            const T* src = static_cast<const T*>(arr == 0 ? r.in[0] : arr == 1 ? r.in[1] : r.in[2]) + (size_t)row * r.L + t;
            cp_async16(st + arr * CS::in + ((size_t)row * kRowE + q * EPC) * sizeof(T), ok ? src : r.in[0], ok ? 16 : 0);
        }
        for (int i = threadIdx.x; i < kTS * (kNP / 4) + kTS / 4; i += kCThreads) {
            if (i < kTS * (kNP / 4)) {
                const int t = ts + i / (kNP / 4), q = i % (kNP / 4);
                const bool ok = t < l1;
                cp_async16(sg + (i / (kNP / 4)) * kGabE + 4 * q, ok ? r.gab + (size_t)t * kNP + 4 * q : r.gab, ok ? 16 : 0);
            } else {
                const int j = i - kTS * (kNP / 4), t = ts + 4 * j;
                const bool ok = t < l1;
                cp_async16(ss + 4 * j, ok ? r.gs + t : r.gs, ok ? 16 : 0);
            }
        }
    } else {
        for (int i = threadIdx.x; i < 3 * kCCh * kTS; i += kCThreads) {
            const int arr = i / (kCCh * kTS), row = (i / kTS) % kCCh, tt = i % kTS;
            const int t = ts + tt;
            const bool ok = row < r.nrows && t < l1;
            T* dst = reinterpret_cast<T*>(st + arr * CS::in) + row * kRowE + tt;
            const T* src = static_cast<const T*>(arr == 0 ? r.in[0] : arr == 1 ? r.in[1] : r.in[2]);
            *dst = ok ? src[(size_t)row * r.L + t] : T(0.0f);
        }
        for (int i = threadIdx.x; i < kTS * kNP + kTS; i += kCThreads) {
            if (i < kTS * kNP) {
                const int t = ts + i / kNP;
                sg[(i / kNP) * kGabE + i % kNP] = t < l1 ? r.gab[(size_t)t * kNP + i % kNP] : 0.0f;
            } else {
                const int t = ts + i - kTS * kNP;
                ss[i - kTS * kNP] = t < l1 ? r.gs[t] : 0.0f;
            }
        }
    }
}

// Two consecutive staged elements as fp32.
__device__ __forceinline__ float2 lds2(const float* q) { return *reinterpret_cast<const float2*>(q); }
__device__ __forceinline__ float2 lds2(const __nv_bfloat16* q) {
    const unsigned w = *reinterpret_cast<const unsigned*>(q);
    return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}
__device__ __forceinline__ void st2v(float* q, float x, float y) {
    __stcs(reinterpret_cast<float2*>(q), make_float2(x, y));
}
__device__ __forceinline__ void st2v(__nv_bfloat16* q, float x, float y) {
    const unsigned w = __bfloat16_as_ushort(__float2bfloat16_rn(x)) |
                       ((unsigned)__bfloat16_as_ushort(__float2bfloat16_rn(y)) << 16);
    __stcs(reinterpret_cast<unsigned*>(q), w);
}

// CTA = kCCh channels of one group of one (b, k) x one span of steps, kSlots
// threads per channel on adjacent lanes; in every group of kCV steps slot q
// takes steps 2q and 2q + 1.  The span streams through kNS shared-memory
// stages of kTS steps (raw, u, gy of the CTA's channels and the group's
// gAbar / M, gs / M).  Each slot keeps its own partial sums of gA, gDskip and
// gbias; the four are added pairwise (the same order in every slot) at the
// end of the span.  Staged steps past the span are zeros and add nothing.
template <typename T, bool VEC>
__global__ void __launch_bounds__(kCThreads, 4) bwd_channel_kernel(const BwdParams p) {
    using CS = ChanStage<T>;
    __shared__ __align__(16) unsigned char smem[kNS * CS::bytes];
    pdl_wait();
    pdl_launch_dependents();
    const int gblk = (p.M + kCCh - 1) / kCCh;  // channel blocks per group
    int bid = blockIdx.x;
    const int span = bid % p.nspan;
    bid /= p.nspan;
    const int jb = bid % gblk;
    bid /= gblk;
    const int g = bid % p.G;
    const int bk = bid / p.G;
    const int b = bk / p.K, k = bk % p.K;
    const int L = p.L, N = p.N;
    const int slot = threadIdx.x % kSlots, ch = threadIdx.x / kSlots;
    const int d0 = g * p.M + jb * kCCh;  // the CTA's first channel
    const int nrows = min(kCCh, p.M - jb * kCCh);
    const bool cv = ch < nrows;
    const int d = d0 + (cv ? ch : 0);
    const size_t seq = (size_t)bk * p.G + g;
    const int c = k * p.D + d;
    const int l0 = span * p.span_len, l1 = min(L, l0 + p.span_len);
    const size_t row0 = ((size_t)bk * p.D + d0) * L;
    ChanRows rows;
    rows.in[0] = static_cast<const T*>(p.raw) + row0;
    rows.in[1] = static_cast<const T*>(p.u) + row0;
    rows.in[2] = static_cast<const T*>(p.gy) + row0;
    rows.gab = p.gab + seq * L * kNP;
    rows.gs = p.gs + seq * L;
    rows.nrows = nrows;
    rows.L = L;
    const size_t row = ((size_t)bk * p.D + d) * L;
    T* gu = static_cast<T*>(p.gu) + row;
    T* graw = static_cast<T*>(p.graw) + row;
    // states as pairs (n, n + 1) for the packed f32x2 operations
    float2 A2[kNP / 2], gA[kNP / 2];
#pragma unroll
    for (int m = 0; m < kNP / 2; ++m) {
        const int n = 2 * m;
        A2[m] = make_float2(n < N ? __ldg(p.A + (size_t)c * N + n) * kLog2e : 0.0f,
                            n + 1 < N ? __ldg(p.A + (size_t)c * N + n + 1) * kLog2e : 0.0f);
        gA[m] = make_float2(0.0f, 0.0f);
    }
    const float bias = __ldg(p.bias + c);
    const float dsk = __ldg(p.Dskip + c);
    const int sp = p.softplus_on;
    float2 gD2 = make_float2(0.0f, 0.0f), gbs2 = make_float2(0.0f, 0.0f);  // per step of the pair
    const int ntile = (l1 - l0 + kTS - 1) / kTS;
#pragma unroll
    for (int j = 0; j < kNS - 1; ++j) {
        if (j < ntile) stage_chan<T, VEC>(smem + j * CS::bytes, rows, l0 + j * kTS, l1);
        cp_async_commit();
    }
    for (int j = 0; j < ntile; ++j) {
        cp_async_wait<kNS - 2>();
        __syncthreads();  // stage j has landed; stage j - 1 is no longer read
        const int jn = j + kNS - 1;
        if (jn < ntile) stage_chan<T, VEC>(smem + (jn % kNS) * CS::bytes, rows, l0 + jn * kTS, l1);
        cp_async_commit();
        const unsigned char* st = smem + (j % kNS) * CS::bytes;
        const float* sgab = reinterpret_cast<const float*>(st + CS::gab);
        const float* sgs = reinterpret_cast<const float*>(st + CS::gs);
        const int ts = l0 + j * kTS;
#pragma unroll
        for (int gi = 0; gi < kTS / kCV; ++gi) {
            const int lt = gi * kCV + 2 * slot;  // this slot's first step in the stage
            const float2 rv = lds2(reinterpret_cast<const T*>(st) + ch * kRowE + lt);
            const float2 uv = lds2(reinterpret_cast<const T*>(st + CS::in) + ch * kRowE + lt);
            const float2 gv = lds2(reinterpret_cast<const T*>(st + 2 * CS::in) + ch * kRowE + lt);
            // the slot's two steps side by side in the packed f32x2 operations
            const float2 v2 = __fadd2_rn(rv, make_float2(bias, bias));
            float2 dl2 = v2, sg2 = make_float2(1.0f, 1.0f);
            if (sp) {
                const float2 e2 = softplus2_e(v2);  // e^-|v|, shared with the derivative
                dl2 = softplus2_from_e(v2, e2);
                const float2 d1 = __fadd2_rn(e2, make_float2(1.0f, 1.0f));
                const float2 r2 = make_float2(rcp(d1.x), rcp(d1.y));
                const float2 er = __fmul2_rn(e2, r2);
                sg2 = make_float2(v2.x >= 0.0f ? r2.x : er.x, v2.y >= 0.0f ? r2.y : er.y);  // softplus'
            }
            const float2 gst2 = *reinterpret_cast<const float2*>(sgs + lt);
            float sum[2];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const float dl = e ? dl2.y : dl2.x;
                const float* w = sgab + (lt + e) * kGabE;
                const float2 dlv = make_float2(dl, dl);
                float2 acc0 = make_float2(0.0f, 0.0f), acc1 = make_float2(0.0f, 0.0f);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float4 w4 = *reinterpret_cast<const float4*>(w + 4 * q);
                    // states (4q, 4q + 1) and (4q + 2, 4q + 3)
                    const float2 x01 = __fmul2_rn(dlv, A2[2 * q]), x23 = __fmul2_rn(dlv, A2[2 * q + 1]);
                    const float2 we01 = __fmul2_rn(make_float2(w4.x, w4.y), make_float2(ex2(x01.x), ex2(x01.y)));
                    const float2 we23 = __fmul2_rn(make_float2(w4.z, w4.w), make_float2(ex2(x23.x), ex2(x23.y)));
                    acc0 = __ffma2_rn(we01, A2[2 * q], acc0);
                    acc1 = __ffma2_rn(we23, A2[2 * q + 1], acc1);
                    gA[2 * q] = __ffma2_rn(we01, dlv, gA[2 * q]);
                    gA[2 * q + 1] = __ffma2_rn(we23, dlv, gA[2 * q + 1]);
                }
                const float2 s2 = __fadd2_rn(acc0, acc1);
                sum[e] = s2.x + s2.y;
            }
            // sum_n gAbar_n A_n e_n / M = ln 2 sum_n (gAbar_n / M) (A_n log2 e) e_n
            const float2 gd2 = __ffma2_rn(gst2, uv, __fmul2_rn(make_float2(sum[0], sum[1]), make_float2(kLn2, kLn2)));
            const float2 gr2 = __fmul2_rn(gd2, sg2);
            const float2 gu2 = __ffma2_rn(make_float2(dsk, dsk), gv, __fmul2_rn(gst2, dl2));
            gD2 = __ffma2_rn(gv, uv, gD2);
            gbs2 = __fadd2_rn(gbs2, gr2);
            const float o_gu[2] = {gu2.x, gu2.y}, o_gr[2] = {gr2.x, gr2.y};
            const int t = ts + lt;
            if (cv) {
                if (VEC) {
                    if (t < l1) {  // l1 is kCV-aligned: both steps or neither
                        st2v(gu + t, o_gu[0], o_gu[1]);
                        st2v(graw + t, o_gr[0], o_gr[1]);
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < 2; ++e) {
                        if (t + e < l1) {
                            gu[t + e] = io<T>::to(o_gu[e]);
                            graw[t + e] = io<T>::to(o_gr[e]);
                        }
                    }
                }
            }
        }
    }
    cp_async_wait<0>();
    float gD = gD2.x + gD2.y, gbs = gbs2.x + gbs2.y;
    // the slots' sums: (s0 + s1) + (s2 + s3) in every slot
#pragma unroll
    for (int m = 1; m < kSlots; m *= 2) {
#pragma unroll
        for (int n = 0; n < kNP / 2; ++n) {
            gA[n].x += __shfl_xor_sync(0xffffffffu, gA[n].x, m);
            gA[n].y += __shfl_xor_sync(0xffffffffu, gA[n].y, m);
        }
        gD += __shfl_xor_sync(0xffffffffu, gD, m);
        gbs += __shfl_xor_sync(0xffffffffu, gbs, m);
    }
    if (slot != 0 || !cv) return;
    const size_t po = ((size_t)b * p.nspan + span) * ((size_t)p.K * p.D) + c;
    float4* pa = reinterpret_cast<float4*>(p.pA + po * kNP);
#pragma unroll
    for (int q = 0; q < kNP / 4; ++q) pa[q] = make_float4(gA[2 * q].x, gA[2 * q].y, gA[2 * q + 1].x, gA[2 * q + 1].y);
    p.pD[po] = gD;
    p.pb[po] = gbs;
}

// ---------------------------------------------------------------- launch 6
// Blocks [0, n_pblk): 32 parameter sums per block, each over the B * nspan
// (batch, span) partials: slice s of 8 adds partials s, s + 8, ... and the
// eight slices are added in slice order (a fixed order).  Blocks from n_pblk
// on: with groups, each (b, k, n, t) of gB and gC summed over the groups in
// group order.
constexpr int kFSlices = 8;
template <typename T>
__global__ void __launch_bounds__(256) bwd_finalize_kernel(const BwdParams p, int n_pblk, long long n_par,
                                                           long long n_bc) {
    __shared__ float part[kFSlices][32];
    pdl_wait();
    pdl_launch_dependents();
    const long long KD = (long long)p.K * p.D;
    if ((int)blockIdx.x < n_pblk) {
        const long long i = (long long)blockIdx.x * 32 + threadIdx.x % 32;  // output: (c, n) of gA, then c, c
        const int sl = threadIdx.x / 32;
        const int np = p.B * p.nspan;
        const float* src = nullptr;
        size_t stride = 0;
        if (i < KD * p.N) {
            src = p.pA + (i / p.N) * kNP + i % p.N;
            stride = (size_t)KD * kNP;
        } else if (i < KD * p.N + KD) {
            src = p.pD + (i - KD * p.N);
            stride = (size_t)KD;
        } else if (i < n_par) {
            src = p.pb + (i - KD * p.N - KD);
            stride = (size_t)KD;
        }
        float s = 0.0f;
        if (src)
            for (int j = sl; j < np; j += kFSlices) s += src[(size_t)j * stride];
        part[sl][threadIdx.x % 32] = s;
        __syncthreads();
        if (sl == 0 && i < n_par) {
            float t = part[0][threadIdx.x];
#pragma unroll
            for (int q = 1; q < kFSlices; ++q) t += part[q][threadIdx.x];
            if (i < KD * p.N)
                p.gA[i] = t;
            else if (i < KD * p.N + KD)
                p.gDskip[i - KD * p.N] = t;
            else
                p.gbias[i - KD * p.N - KD] = t;
        }
        return;
    }
    const long long j = (long long)(blockIdx.x - n_pblk) * 256 + threadIdx.x;
    if (p.G > 1 && j < n_bc) {
        // (bk, n, t) of gB and gC
        const long long t = j % p.L, n = (j / p.L) % p.N, bk = j / ((long long)p.L * p.N);
        float sb = 0.0f, sc = 0.0f;
        for (int g = 0; g < p.G; ++g) {
            const size_t w = (((size_t)bk * p.G + g) * kNP + n) * p.L + t;
            sb += p.gBw[w];
            sc += p.gCw[w];
        }
        static_cast<T*>(p.gB)[j] = io<T>::to(sb);
        static_cast<T*>(p.gC)[j] = io<T>::to(sc);
    }
}

bool aligned_to(const void* q, size_t a) { return reinterpret_cast<uintptr_t>(q) % a == 0; }

template <typename T>
vmb_status launch_t(const BwdParams& p, cudaStream_t stream) {
    const long long S = (long long)p.B * p.K * p.G;
    const long long nlb = (p.L + kRT - 1) / kRT;
    const long long n_pairs = S * p.nch;
    const long long g5 = (long long)p.B * p.K * p.G * ((p.M + kCCh - 1) / kCCh) * p.nspan;
    if (S * nlb > INT32_MAX || n_pairs > INT32_MAX || S * 32 > INT32_MAX || g5 > INT32_MAX ||
        (long long)p.D * p.L > INT32_MAX)
        return VMB_ERR_UNSUPPORTED;
    BwdParams q = p;
    void* a1[] = {&q};
    const void* k1 = p.saved ? reinterpret_cast<const void*>(&bwd_gysum_kernel<T>)
                             : reinterpret_cast<const void*>(&bwd_reduce_kernel<T>);
    if (launch_kernel(k1, dim3((unsigned)(S * nlb)), dim3(kRThreads), 0, a1, stream) != cudaSuccess)
        return VMB_ERR_CUDA;
    int np = (int)n_pairs;
    void* a2[] = {&q, &np};
    const unsigned g2 = (unsigned)((n_pairs + kSWarps - 1) / kSWarps);
    if (launch_kernel(reinterpret_cast<const void*>(&bwd_summary_kernel<T>), dim3(g2), dim3(32 * kSWarps), 0, a2,
                      stream) != cudaSuccess)
        return VMB_ERR_CUDA;
    int nl = (int)(S * 32);
    void* a3[] = {&q, &nl};
    if (launch_kernel(reinterpret_cast<const void*>(&bwd_carry_kernel), dim3((unsigned)((nl + 255) / 256)), dim3(256),
                      0, a3, stream) != cudaSuccess)
        return VMB_ERR_CUDA;
    if (launch_kernel(reinterpret_cast<const void*>(&bwd_chunk_kernel<T>), dim3(g2), dim3(32 * kSWarps), 0, a2,
                      stream) != cudaSuccess)
        return VMB_ERR_CUDA;
    // async copies: rows, spans and the end kCV-aligned, inputs 16-byte aligned, pairs of outputs aligned
    const bool vec = p.L % kCV == 0 && aligned_to(p.u, 16) && aligned_to(p.raw, 16) && aligned_to(p.gy, 16) &&
                     aligned_to(p.gu, 2 * sizeof(T)) && aligned_to(p.graw, 2 * sizeof(T));
    const void* k5 = vec ? reinterpret_cast<const void*>(&bwd_channel_kernel<T, true>)
                         : reinterpret_cast<const void*>(&bwd_channel_kernel<T, false>);
    if (launch_kernel(k5, dim3((unsigned)g5), dim3(kCThreads), 0, a1, stream) != cudaSuccess) return VMB_ERR_CUDA;
    long long n_par = (long long)p.K * p.D * (p.N + 2);
    long long n_bc = p.G > 1 ? (long long)p.B * p.K * p.N * p.L : 0;
    const long long pblk = (n_par + 31) / 32;
    const long long g6 = pblk + (n_bc + 255) / 256;
    if (g6 > INT32_MAX) return VMB_ERR_UNSUPPORTED;
    int n_pblk = (int)pblk;
    void* a6[] = {&q, &n_pblk, &n_par, &n_bc};
    return launch_kernel(reinterpret_cast<const void*>(&bwd_finalize_kernel<T>), dim3((unsigned)g6), dim3(256), 0, a6,
                         stream) == cudaSuccess
               ? VMB_OK
               : VMB_ERR_CUDA;
}

}  // namespace

size_t mean_bwd_workspace_bytes(long long B, long long K, long long D, long long N, long long L, long long G) {
    return bwd_layout(B, K, D, N, L, G).total;
}

vmb_status launch_mean_bwd(const MeanBwdArgs& a, cudaStream_t stream) {
    BwdParams p{};
    p.u = a.u;
    p.raw = a.delta;
    p.A = a.A;
    p.Bs = a.Bs;
    p.Cs = a.Cs;
    p.Dskip = a.Dskip;
    p.bias = a.bias;
    p.gy = a.gy;
    p.gu = a.gu;
    p.graw = a.gdelta;
    p.gA = a.gA;
    p.gB = a.gBs;
    p.gC = a.gCs;
    p.gDskip = a.gDskip;
    p.gbias = a.gbias;
    p.B = a.B;
    p.K = a.K;
    p.D = a.D;
    p.N = a.N;
    p.L = a.L;
    p.G = a.groups;
    p.M = a.D / a.groups;
    p.softplus_on = (a.flags & VMB_FLAG_SOFTPLUS) ? 1 : 0;
    const BwdLayout w = bwd_layout(a.B, a.K, a.D, a.N, a.L, a.groups);
    p.nch = w.nch;
    p.nspan = w.nspan;
    p.span_len = w.span_len;
    unsigned char* ws = static_cast<unsigned char*>(a.ws);
    p.ms = a.saved ? const_cast<float*>(a.saved) : reinterpret_cast<float*>(ws + w.ms);
    p.saved = a.saved != nullptr;
    {
        const size_t bal = a.dtype == VMB_BF16 ? 8 : 16;
        // (the caller's saved means need only 4-byte alignment)
        p.vec = (a.L % 4 == 0 && reinterpret_cast<uintptr_t>(a.Bs) % bal == 0 &&
                 reinterpret_cast<uintptr_t>(a.Cs) % bal == 0 && reinterpret_cast<uintptr_t>(p.ms) % 16 == 0)
                    ? 1
                    : 0;
    }
    p.gyb = reinterpret_cast<float*>(ws + w.gyb);
    p.sumP = reinterpret_cast<float*>(ws + w.sumP);
    p.sumH = reinterpret_cast<float*>(ws + w.sumH);
    p.sumV = reinterpret_cast<float*>(ws + w.sumV);
    p.gab = reinterpret_cast<float*>(ws + w.gab);
    p.gs = reinterpret_cast<float*>(ws + w.gs);
    p.gBw = reinterpret_cast<float*>(ws + w.gBw);
    p.gCw = reinterpret_cast<float*>(ws + w.gCw);
    p.pA = reinterpret_cast<float*>(ws + w.pA);
    p.pD = reinterpret_cast<float*>(ws + w.pD);
    p.pb = reinterpret_cast<float*>(ws + w.pb);
    return a.dtype == VMB_BF16 ? launch_t<__nv_bfloat16>(p, stream) : launch_t<float>(p, stream);
}

}  // namespace vmb
