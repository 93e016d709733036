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
// Four launches, every reduction in a fixed order (results are deterministic):
//   1. per (sequence, step): the group means Abar, sm and the summed output
//      gradient gyb (a thread per step, the group's channels split in two);
//   2. per sequence: the states forward, then the adjoint recurrence backward
//      (a half warp per sequence, a lane per state; gs reduced over the lanes);
//   3. per channel: the chain rule through the mean and the softplus, gu and
//      graw, and per-batch partial sums of gA, gDskip and gbias;
//   4. the partial sums added over the batch (and gB, gC over the groups).
#include <mutex>

#include "vmb_common.cuh"
#include "vmb_internal.h"

namespace vmb {
namespace {

constexpr int kNP = 16;       // states per sequence as stored (N <= 16, zero padded)
constexpr int kRT = 128;      // steps per CTA of launch 1
constexpr int kRThreads = 256;
constexpr int kCThreads = 128;  // channels per CTA of launch 3
constexpr int kCT = 4;          // steps per iteration of launch 3

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
    // workspace arrays (fp32)
    float* abar;  // [S][L][kNP]
    float* sm;    // [S][L]
    float* gyb;   // [S][L]
    float* hst;   // [S][L + 1][kNP]: h(t - 1) at row t
    float* gab;   // [S][L][kNP]
    float* gs;    // [S][L]
    float* gBw;   // [S][kNP][L] (groups > 1): per-group contributions to gB
    float* gCw;   // [S][kNP][L]
    float* pA;    // [B][K D][kNP] per-batch partial sums
    float* pD;    // [B][K D]
    float* pb;    // [B][K D]
};

// Workspace layout (256-byte aligned arrays).
struct BwdLayout {
    size_t abar, sm, gyb, hst, gab, gs, gBw, gCw, pA, pD, pb, total;
};
BwdLayout bwd_layout(long long B, long long K, long long D, long long L, long long G) {
    const long long S = B * K * G;
    BwdLayout w{};
    size_t o = 0;
    auto take = [&](size_t bytes) {
        const size_t at = o;
        o = align_up(o + bytes, 256);
        return at;
    };
    w.abar = take((size_t)S * L * kNP * 4);
    w.sm = take((size_t)S * L * 4);
    w.gyb = take((size_t)S * L * 4);
    w.hst = take((size_t)S * (L + 1) * kNP * 4);
    w.gab = take((size_t)S * L * kNP * 4);
    w.gs = take((size_t)S * L * 4);
    w.gBw = take(G > 1 ? (size_t)S * kNP * L * 4 : 0);
    w.gCw = take(G > 1 ? (size_t)S * kNP * L * 4 : 0);
    w.pA = take((size_t)B * K * D * kNP * 4);
    w.pD = take((size_t)B * K * D * 4);
    w.pb = take((size_t)B * K * D * 4);
    w.total = o;
    return w;
}

__device__ __forceinline__ float delta_of(float v, int softplus_on) { return softplus_on ? softplus(v) : v; }

// softplus'(v) = the logistic function 1 / (1 + e^-v), from e^-|v| (no overflow)
__device__ __forceinline__ float softplus_grad(float v) {
    const float e = ex2(-fabsf(v) * kLog2e);
    const float r = 1.0f / (1.0f + e);
    return v >= 0.0f ? r : e * r;
}

// ---------------------------------------------------------------- launch 1
// CTA = one sequence x kRT steps; thread (t, half) sums its half of the
// group's channels at step t; the two halves are added in shared memory.
template <typename T>
__global__ void __launch_bounds__(kRThreads) bwd_reduce_kernel(const BwdParams p) {
    pdl_wait();
    pdl_launch_dependents();
    __shared__ float red[2][kNP + 2][kRT];
    const int nlb = (p.L + kRT - 1) / kRT;
    const int seq = blockIdx.x / nlb;  // (b, k, g)
    const int t = (blockIdx.x % nlb) * kRT + threadIdx.x % kRT;
    const int half = threadIdx.x / kRT;
    const int b = seq / (p.K * p.G), k = (seq / p.G) % p.K, g = seq % p.G;
    const bool tv = t < p.L;
    const int L = p.L, N = p.N, M = p.M;
    const size_t row0 = ((size_t)b * p.K + k) * p.D + (size_t)g * M;  // first (b, k, d) row of the group
    const T* u = static_cast<const T*>(p.u) + row0 * L;
    const T* raw = static_cast<const T*>(p.raw) + row0 * L;
    const T* gy = static_cast<const T*>(p.gy) + row0 * L;
    float acc[kNP];
#pragma unroll
    for (int n = 0; n < kNP; ++n) acc[n] = 0.0f;
    float su = 0.0f, sg = 0.0f;
    if (tv) {
        for (int j = half; j < M; j += 2) {
            const int c = k * p.D + g * M + j;
            const float v = io<T>::ld(raw + (size_t)j * L + t) + __ldg(p.bias + c);
            const float dl = delta_of(v, p.softplus_on);
            const float dl2 = dl * kLog2e;
            const float* Ac = p.A + (size_t)c * N;
#pragma unroll
            for (int n = 0; n < kNP; ++n)
                if (n < N) acc[n] += ex2(dl2 * __ldg(Ac + n));
            su = fmaf(dl, io<T>::ld(u + (size_t)j * L + t), su);
            sg += io<T>::ld(gy + (size_t)j * L + t);
        }
    }
    const int tt = threadIdx.x % kRT;
#pragma unroll
    for (int n = 0; n < kNP; ++n) red[half][n][tt] = acc[n];
    red[half][kNP][tt] = su;
    red[half][kNP + 1][tt] = sg;
    __syncthreads();
    if (half == 0 && tv) {
        const float inv = 1.0f / (float)M;
        float* ab = p.abar + ((size_t)seq * L + t) * kNP;
#pragma unroll
        for (int n = 0; n < kNP; ++n) ab[n] = (red[0][n][tt] + red[1][n][tt]) * inv;
        p.sm[(size_t)seq * L + t] = (red[0][kNP][tt] + red[1][kNP][tt]) * inv;
        p.gyb[(size_t)seq * L + t] = red[0][kNP + 1][tt] + red[1][kNP + 1][tt];
    }
}

// ---------------------------------------------------------------- launch 2
// A half warp per sequence, lane n owns state n: the states forward, then the
// adjoint recurrence backward in time.
template <typename T>
__global__ void __launch_bounds__(128) bwd_scan_kernel(const BwdParams p, int n_seq) {
    pdl_wait();
    pdl_launch_dependents();
    const int seq = (blockIdx.x * 128 + threadIdx.x) / kNP;
    const int n = threadIdx.x % kNP;
    const bool sv = seq < n_seq;
    const int L = p.L, N = p.N;
    const int bk = sv ? seq / p.G : 0;
    const bool nv = sv && n < N;
    const T* Bn = static_cast<const T*>(p.Bs) + ((size_t)bk * N + (nv ? n : 0)) * L;
    const T* Cn = static_cast<const T*>(p.Cs) + ((size_t)bk * N + (nv ? n : 0)) * L;
    const size_t sq = sv ? (size_t)seq : 0;
    const float* ab = p.abar + sq * L * kNP + n;
    const float* smv = p.sm + sq * L;
    const float* gybv = p.gyb + sq * L;
    float* hs = p.hst + sq * (size_t)(L + 1) * kNP + n;
    float* ga = p.gab + sq * L * kNP + n;
    // forward: hst row t holds h(t - 1)
    float h = 0.0f;
    if (sv) hs[0] = 0.0f;
    for (int t = 0; t < L; ++t) {
        const float bt = nv ? io<T>::ld(Bn + t) : 0.0f;
        h = sv ? fmaf(ab[(size_t)t * kNP], h, bt * smv[t]) : 0.0f;
        if (sv) hs[(size_t)(t + 1) * kNP] = h;
    }
    // backward: lam_n(t) = C_n(t) gyb(t) + Abar_n(t+1) lam_n(t+1)
    float lam = 0.0f;
    T* gBo = static_cast<T*>(p.gB) + ((size_t)bk * N + (nv ? n : 0)) * L;
    T* gCo = static_cast<T*>(p.gC) + ((size_t)bk * N + (nv ? n : 0)) * L;
    float* gBw = p.gBw + (sq * kNP + n) * L;
    float* gCw = p.gCw + (sq * kNP + n) * L;
    for (int t = L - 1; t >= 0; --t) {
        const float gyt = sv ? gybv[t] : 0.0f;
        const float ct = nv ? io<T>::ld(Cn + t) : 0.0f;
        const float bt = nv ? io<T>::ld(Bn + t) : 0.0f;
        lam = fmaf(ct, gyt, lam);
        const float ht = sv ? hs[(size_t)(t + 1) * kNP] : 0.0f;
        const float hprev = sv ? hs[(size_t)t * kNP] : 0.0f;
        const float gc = gyt * ht, gb = lam * (sv ? smv[t] : 0.0f);
        if (nv) {
            if (p.G == 1) {
                gCo[t] = io<T>::to(gc);
                gBo[t] = io<T>::to(gb);
            } else {
                gCw[t] = gc;
                gBw[t] = gb;
            }
        }
        if (sv) ga[(size_t)t * kNP] = nv ? lam * hprev : 0.0f;
        // gs(t) = sum over the half warp's lanes of lam_n B_n(t), in a fixed order
        float part = nv ? lam * bt : 0.0f;
#pragma unroll
        for (int m = 8; m >= 1; m >>= 1) part += __shfl_xor_sync(0xffffffffu, part, m);
        if (sv && n == 0) p.gs[sq * L + t] = part;
        lam = sv ? lam * ab[(size_t)t * kNP] : 0.0f;
    }
}

// ---------------------------------------------------------------- launch 3
// CTA = kCThreads channels of one sequence's direction block; thread = one
// channel, walking its row kCT steps at a time; gAbar and gs of those steps
// are staged in shared memory (one per sequence group of the CTA's channels).
template <typename T>
__global__ void __launch_bounds__(kCThreads) bwd_channel_kernel(const BwdParams p) {
    pdl_wait();
    pdl_launch_dependents();
    const int dblk = (p.D + kCThreads - 1) / kCThreads;
    const int bk = blockIdx.x / dblk;
    const int d = (blockIdx.x % dblk) * kCThreads + threadIdx.x;
    const bool dv = d < p.D;
    const int b = bk / p.K, k = bk % p.K;
    const int L = p.L, N = p.N, M = p.M;
    const int g = dv ? d / M : 0;
    const size_t seq = (size_t)bk * p.G + g;
    const int c = k * p.D + (dv ? d : 0);
    const size_t row = (size_t)bk * p.D + (dv ? d : 0);
    const T* u = static_cast<const T*>(p.u) + row * L;
    const T* raw = static_cast<const T*>(p.raw) + row * L;
    const T* gy = static_cast<const T*>(p.gy) + row * L;
    T* gu = static_cast<T*>(p.gu) + row * L;
    T* graw = static_cast<T*>(p.graw) + row * L;
    const float* gab = p.gab + seq * L * kNP;
    const float* gsv = p.gs + seq * L;
    float A[kNP], A2[kNP], gA[kNP];
#pragma unroll
    for (int n = 0; n < kNP; ++n) {
        A[n] = (dv && n < N) ? __ldg(p.A + (size_t)c * N + n) : 0.0f;
        A2[n] = A[n] * kLog2e;
        gA[n] = 0.0f;
    }
    const float bias = dv ? __ldg(p.bias + c) : 0.0f;
    const float dsk = dv ? __ldg(p.Dskip + c) : 0.0f;
    const float invM = 1.0f / (float)M;
    float gD = 0.0f, gbs = 0.0f;
    if (dv) {
        for (int t = 0; t < L; ++t) {
            const float v = io<T>::ld(raw + t) + bias;
            const float dl = delta_of(v, p.softplus_on);
            const float uu = io<T>::ld(u + t), gyy = io<T>::ld(gy + t);
            const float gst = gsv[t];
            const float4* ga4 = reinterpret_cast<const float4*>(gab + (size_t)t * kNP);
            float gd = gst * uu;
#pragma unroll
            for (int q = 0; q < kNP / 4; ++q) {
                const float4 w = ga4[q];
                const float wv[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int n = 4 * q + i;
                    const float e = ex2(dl * A2[n]);
                    const float we = wv[i] * e;
                    gd = fmaf(we, A[n], gd);
                    gA[n] = fmaf(we, dl, gA[n]);
                }
            }
            gd *= invM;
            const float gv = p.softplus_on ? gd * softplus_grad(v) : gd;
            gu[t] = io<T>::to(fmaf(dsk, gyy, gst * dl * invM));
            graw[t] = io<T>::to(gv);
            gD = fmaf(gyy, uu, gD);
            gbs += gv;
        }
        float* pa = p.pA + ((size_t)b * p.K * p.D + c) * kNP;
#pragma unroll
        for (int n = 0; n < kNP; ++n) pa[n] = gA[n] * invM;
        p.pD[(size_t)b * p.K * p.D + c] = gD;
        p.pb[(size_t)b * p.K * p.D + c] = gbs;
    }
}

// ---------------------------------------------------------------- launch 4
// The per-batch partial sums added in batch order; with groups, each
// (b, k, n, t) of gB and gC summed over the groups in group order.
template <typename T>
__global__ void __launch_bounds__(256) bwd_finalize_kernel(const BwdParams p, long long n_par, long long n_bc) {
    pdl_wait();
    pdl_launch_dependents();
    const long long i = (long long)blockIdx.x * 256 + threadIdx.x;
    const long long KD = (long long)p.K * p.D;
    if (i < n_par) {
        // i over (c, n) for gA, then c for gDskip, then c for gbias
        if (i < KD * p.N) {
            const long long c = i / p.N, n = i % p.N;
            float s = 0.0f;
            for (int b = 0; b < p.B; ++b) s += p.pA[((size_t)b * KD + c) * kNP + n];
            p.gA[i] = s;
        } else if (i < KD * p.N + KD) {
            const long long c = i - KD * p.N;
            float s = 0.0f;
            for (int b = 0; b < p.B; ++b) s += p.pD[(size_t)b * KD + c];
            p.gDskip[c] = s;
        } else {
            const long long c = i - KD * p.N - KD;
            float s = 0.0f;
            for (int b = 0; b < p.B; ++b) s += p.pb[(size_t)b * KD + c];
            p.gbias[c] = s;
        }
    } else if (p.G > 1 && i < n_par + n_bc) {
        // (bk, n, t) of gB and gC
        const long long j = i - n_par;
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

template <typename T>
vmb_status launch_t(const BwdParams& p, cudaStream_t stream) {
    const long long S = (long long)p.B * p.K * p.G;
    const long long nlb = (p.L + kRT - 1) / kRT;
    if (S * nlb > INT32_MAX) return VMB_ERR_UNSUPPORTED;
    BwdParams q = p;
    void* a1[] = {&q};
    if (launch_kernel(reinterpret_cast<const void*>(&bwd_reduce_kernel<T>), dim3((unsigned)(S * nlb)), dim3(kRThreads),
                      0, a1, stream) != cudaSuccess)
        return VMB_ERR_CUDA;
    int n_seq = (int)S;
    void* a2[] = {&q, &n_seq};
    const unsigned g2 = (unsigned)((S * kNP + 127) / 128);
    if (launch_kernel(reinterpret_cast<const void*>(&bwd_scan_kernel<T>), dim3(g2), dim3(128), 0, a2, stream) !=
        cudaSuccess)
        return VMB_ERR_CUDA;
    const long long g3 = (long long)p.B * p.K * ((p.D + kCThreads - 1) / kCThreads);
    if (g3 > INT32_MAX) return VMB_ERR_UNSUPPORTED;
    if (launch_kernel(reinterpret_cast<const void*>(&bwd_channel_kernel<T>), dim3((unsigned)g3), dim3(kCThreads), 0,
                      a1, stream) != cudaSuccess)
        return VMB_ERR_CUDA;
    long long n_par = (long long)p.K * p.D * (p.N + 2);
    long long n_bc = p.G > 1 ? (long long)p.B * p.K * p.N * p.L : 0;
    const long long g4 = (n_par + n_bc + 255) / 256;
    if (g4 > INT32_MAX) return VMB_ERR_UNSUPPORTED;
    void* a4[] = {&q, &n_par, &n_bc};
    return launch_kernel(reinterpret_cast<const void*>(&bwd_finalize_kernel<T>), dim3((unsigned)g4), dim3(256), 0, a4,
                         stream) == cudaSuccess
               ? VMB_OK
               : VMB_ERR_CUDA;
}

}  // namespace

size_t mean_bwd_workspace_bytes(long long B, long long K, long long D, long long L, long long G) {
    return bwd_layout(B, K, D, L, G).total;
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
    const BwdLayout w = bwd_layout(a.B, a.K, a.D, a.L, a.groups);
    unsigned char* ws = static_cast<unsigned char*>(a.ws);
    p.abar = reinterpret_cast<float*>(ws + w.abar);
    p.sm = reinterpret_cast<float*>(ws + w.sm);
    p.gyb = reinterpret_cast<float*>(ws + w.gyb);
    p.hst = reinterpret_cast<float*>(ws + w.hst);
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
