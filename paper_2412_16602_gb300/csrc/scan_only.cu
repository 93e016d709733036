// scan_only.cu - the paper's own kernel setting (Sec. 4, "Kernel
// Implementation"): the discretisation runs before the scan, and the scan
// kernel reads the materialised operands Abar = exp(delta A) and Bbar u
// ([B][K][D][N][L], or [B][K][1][N][L] after the channel mean of Eq. 9).
//
//   discretise_kernel       Eqs. 4, 6 for every (b, k, d, n, l), fp32 out
//   discretise_mean_kernel  Eq. 9's T on the discretised operands: the means
//                           over the D channels of each (b, k), fp32 out
//   scan_only_kernel        Eq. 3 without the skip term on the materialised
//                           operands: h_n = dA h_n + dBu, y = sum_n C_n h_n
//
// The fused kernels of full_scan.cu / mean_scan.cu are the product path; these
// exist to measure the split the paper timed (its Tables 1 and 2) on GB300.
#include <stdint.h>

#include "vmb_common.cuh"
#include "vmb_internal.h"

namespace vmb {
namespace {

constexpr int kDiscThreads = 256;

struct DiscParams {
    const void* u;
    const void* dl;
    const float* A;
    const void* Bs;
    const float* bias;
    float* dA;
    float* dBu;
    int K, D, N, L;
    int nlb;  // L blocks per row (discretise) or per (b, k) (mean)
    int softplus_on;
};

// Eq. 4 for one (delta, A, B, u): the decay and the input term, in the same
// operation order as the fused scans (Euler: (delta u) B; zero-order hold:
// ((e^{delta A} - 1) / A) B u, delta B u at A = 0).
template <bool ZOH>
__device__ __forceinline__ void disc_one(float dlt, float a, float a2, float b, float uu, float& da, float& dbu) {
    if constexpr (ZOH) {
        const float em1 = expm1f(dlt * a);
        da = 1.0f + em1;
        dbu = (a != 0.0f ? em1 / a : dlt) * b * uu;
    } else {
        da = ex2(dlt * a2);
        dbu = (dlt * uu) * b;
    }
}

// One thread per (row, l), row = (b, k, d); the N states of the step are
// written to N rows of the [row][N][L] output, each store coalesced over l.
template <typename T, bool ZOH>
__global__ void __launch_bounds__(kDiscThreads) discretise_kernel(const DiscParams p) {
    pdl_wait();
    pdl_launch_dependents();
    const long long row = blockIdx.x / p.nlb;
    const int l = (int)(blockIdx.x % p.nlb) * kDiscThreads + threadIdx.x;
    if (l >= p.L) return;
    const int d = (int)(row % p.D);
    const long long bk = row / p.D;
    const int k = (int)(bk % p.K);
    const int c = k * p.D + d;
    const size_t e = (size_t)row * p.L + l;
    const float v = io<T>::ld(static_cast<const T*>(p.dl) + e) + p.bias[c];
    const float dlt = p.softplus_on ? softplus(v) : v;
    const float uu = io<T>::ld(static_cast<const T*>(p.u) + e);
    const T* bs = static_cast<const T*>(p.Bs) + (size_t)bk * p.N * p.L + l;
    const float* Ac = p.A + (size_t)c * p.N;
    float* oa = p.dA + (size_t)row * p.N * p.L + l;
    float* ob = p.dBu + (size_t)row * p.N * p.L + l;
    for (int n = 0; n < p.N; ++n) {
        const float a = Ac[n];
        float da, dbu;
        disc_one<ZOH>(dlt, a, a * kLog2e, io<T>::ld(bs + (size_t)n * p.L), uu, da, dbu);
        oa[(size_t)n * p.L] = da;
        ob[(size_t)n * p.L] = dbu;
    }
}

// Channel means of the discretised operands.  A CTA covers 32 consecutive
// steps of one (b, k); its 8 warps take every 8th channel, each lane one step,
// and the 8 partial sums are added in warp order (a fixed order, so the
// result does not depend on scheduling).  Euler: the mean of delta_d u_d B_n
// is B_n times the mean of delta_d u_d; zero-order hold keeps one sum of
// ((e^{delta A} - 1) / A) u per state and multiplies by B_n at the end.
constexpr int kMeanSteps = 32;
constexpr int kMeanGroups = kDiscThreads / kMeanSteps;

template <typename T, bool ZOH>
__global__ void __launch_bounds__(kDiscThreads) discretise_mean_kernel(const DiscParams p) {
    pdl_wait();
    pdl_launch_dependents();
    __shared__ float sa[kMeanGroups][16][kMeanSteps];
    __shared__ float sb[kMeanGroups][16][kMeanSteps];
    const long long bk = blockIdx.x / p.nlb;
    const int lane = threadIdx.x % kMeanSteps, grp = threadIdx.x / kMeanSteps;
    const int l = (int)(blockIdx.x % p.nlb) * kMeanSteps + lane;
    const bool lv = l < p.L;
    const int k = (int)(bk % p.K);
    const int N = p.N;
    float acc[16], accb[16];
#pragma unroll
    for (int n = 0; n < 16; ++n) acc[n] = accb[n] = 0.0f;
    if (lv) {
        for (int d = grp; d < p.D; d += kMeanGroups) {
            const int c = k * p.D + d;
            const size_t e = ((size_t)bk * p.D + d) * p.L + l;
            const float v = io<T>::ld(static_cast<const T*>(p.dl) + e) + p.bias[c];
            const float dlt = p.softplus_on ? softplus(v) : v;
            const float uu = io<T>::ld(static_cast<const T*>(p.u) + e);
            const float* Ac = p.A + (size_t)c * N;
            if constexpr (!ZOH) accb[0] = fmaf(dlt, uu, accb[0]);
#pragma unroll
            for (int n = 0; n < 16; ++n) {
                if (n < N) {
                    const float a = Ac[n];
                    if constexpr (ZOH) {
                        const float em1 = expm1f(dlt * a);
                        acc[n] += 1.0f + em1;
                        accb[n] = fmaf(a != 0.0f ? em1 / a : dlt, uu, accb[n]);
                    } else {
                        acc[n] += ex2(dlt * (a * kLog2e));
                    }
                }
            }
        }
    }
#pragma unroll
    for (int n = 0; n < 16; ++n) {
        sa[grp][n][lane] = acc[n];
        sb[grp][n][lane] = accb[n];
    }
    __syncthreads();
    const float inv = 1.0f / (float)p.D;
    // thread (n, step) finishes state n of step `lane` for n = grp, grp + 8
    for (int n = grp; n < N; n += kMeanGroups) {
        float s = 0.0f, t = 0.0f;
#pragma unroll
        for (int g = 0; g < kMeanGroups; ++g) {
            s += sa[g][n][lane];
            t += sb[g][ZOH ? n : 0][lane];
        }
        if (lv) {
            const size_t o = ((size_t)bk * N + n) * p.L + l;
            const float b = io<T>::ld(static_cast<const T*>(p.Bs) + o);
            p.dA[o] = s * inv;
            p.dBu[o] = (t * inv) * b;
        }
    }
}

// ----------------------------------------------------------------- scan alone
// A CTA owns one channel.  Its L steps are cut into S segments; lane (s, n)
// scans state n over segment s twice: first from zero, giving the segment's
// decay product P and end state H, then from its carry, producing the output.
// The carries are an exclusive scan over the segments of the affine maps
// h -> P h + H (composition (P1, H1) then (P2, H2) = (P2 P1, P2 H1 + H2)), done
// in shared memory in log2(S) rounds (Hillis-Steele: a fixed order, so the
// result is reproducible).  A channel's operands (N L floats each) are small
// enough, and few enough CTAs are resident, that the second pass reads them
// from L2.  The NP lanes of one segment are adjacent, and y = sum_n C_n h_n is
// reduced over them every 8 steps by a transposed butterfly.
struct OnlyParams {
    const float* dA;
    const float* dBu;
    const void* Cs;
    float* y;
    long long channels;  // B * K * Dm
    int Dm, N, L;
    int seg_len;  // steps per segment, a multiple of 8
    int vec;      // rows 32-byte aligned at every 8-step block
};

template <int NP>
struct OnlyShape {
    static constexpr int S = NP >= 4 ? 64 : 256 / NP;  // segments per channel
    static constexpr int THREADS = S * NP;             // 1024, 512 or 256
};

template <typename T>
__device__ __forceinline__ void load8(const T* p, int t, int t1, bool vec, float (&v)[8], float fill) {
    if (vec && t + 8 <= t1) {
        if constexpr (sizeof(T) == 4) {
            const float4 a = __ldg(reinterpret_cast<const float4*>(p + t));
            const float4 b = __ldg(reinterpret_cast<const float4*>(p + t) + 1);
            v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
            v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
        } else {
            const uint4 q = __ldg(reinterpret_cast<const uint4*>(p + t));
            const __nv_bfloat16* h = reinterpret_cast<const __nv_bfloat16*>(&q);
#pragma unroll
            for (int j = 0; j < 8; ++j) v[j] = __bfloat162float(h[j]);
        }
    } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) v[j] = (t + j < t1) ? io<T>::ld(p + t + j) : fill;
    }
}

// v[0..8) summed over the NP adjacent lanes; afterwards the lane with index
// r (0 <= r < NP) in its group holds the sums for steps base(r) ..
// base(r) + 8 / min(NP, 8) - 1 in v[0..), with NP = 16 lane pairs sharing a step.
template <int NP>
__device__ __forceinline__ void reduce8(float (&v)[8], int r) {
    if constexpr (NP >= 16) {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const bool up = (r & 8) != 0;
            const float keep = up ? v[i + 4] : v[i], send = up ? v[i] : v[i + 4];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
        }
    }
    if constexpr (NP >= 8) {
        constexpr int CNT = NP >= 16 ? 4 : 8;
#pragma unroll
        for (int i = 0; i < CNT / 2; ++i) {
            const bool up = (r & 4) != 0;
            const float keep = up ? v[i + CNT / 2] : v[i], send = up ? v[i] : v[i + CNT / 2];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
        }
    }
    if constexpr (NP >= 4) {
        constexpr int CNT = NP >= 16 ? 2 : (NP >= 8 ? 4 : 8);
#pragma unroll
        for (int i = 0; i < CNT / 2; ++i) {
            const bool up = (r & 2) != 0;
            const float keep = up ? v[i + CNT / 2] : v[i], send = up ? v[i] : v[i + CNT / 2];
            v[i] = keep + __shfl_xor_sync(0xffffffffu, send, 2);
        }
    }
    if constexpr (NP >= 2) {
        constexpr int CNT = NP >= 16 ? 1 : (NP >= 8 ? 2 : (NP >= 4 ? 4 : 8));
        if constexpr (CNT == 1) {
            v[0] += __shfl_xor_sync(0xffffffffu, v[0], 1);
        } else {
#pragma unroll
            for (int i = 0; i < CNT / 2; ++i) {
                const bool up = (r & 1) != 0;
                const float keep = up ? v[i + CNT / 2] : v[i], send = up ? v[i] : v[i + CNT / 2];
                v[i] = keep + __shfl_xor_sync(0xffffffffu, send, 1);
            }
        }
    }
}

template <typename T, int NP>
__global__ void __launch_bounds__(OnlyShape<NP>::THREADS) scan_only_kernel(const OnlyParams p) {
    pdl_wait();
    pdl_launch_dependents();
    constexpr int S = OnlyShape<NP>::S;
    __shared__ float sP[S][NP], sH[S][NP];
    const int n = threadIdx.x % NP;
    const int s = threadIdx.x / NP;
    const long long ch = blockIdx.x;
    const bool nv = n < p.N;
    const long long bk = ch / p.Dm;
    const int t0 = min(p.L, s * p.seg_len), t1 = min(p.L, t0 + p.seg_len);
    const float* ra = p.dA + ((size_t)ch * p.N + (nv ? n : 0)) * p.L;
    const float* rb = p.dBu + ((size_t)ch * p.N + (nv ? n : 0)) * p.L;
    const T* rc = static_cast<const T*>(p.Cs) + ((size_t)bk * p.N + (nv ? n : 0)) * p.L;
    const bool vec = p.vec != 0;
    // pass 1: the segment from a zero state
    float P = 1.0f, H = 0.0f;
    if (nv) {
        for (int t = t0; t < t1; t += 8) {
            float a[8], b[8];
            load8<float>(ra, t, t1, vec, a, 1.0f);
            load8<float>(rb, t, t1, vec, b, 0.0f);
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                P *= a[j];
                H = fmaf(a[j], H, b[j]);
            }
        }
    }
    sP[s][n] = P;
    sH[s][n] = H;
    __syncthreads();
    // inclusive scan over the segments (earlier segment applied first)
#pragma unroll 1
    for (int off = 1; off < S; off <<= 1) {
        float pp = 1.0f, hh = 0.0f;
        if (s >= off) {
            pp = sP[s - off][n];
            hh = sH[s - off][n];
        }
        __syncthreads();
        if (s >= off) {
            H = fmaf(P, hh, H);
            P *= pp;
            sP[s][n] = P;
            sH[s][n] = H;
        }
        __syncthreads();
    }
    float h = (nv && s > 0) ? sH[s - 1][n] : 0.0f;  // carry into this segment
    float* yr = p.y + (size_t)ch * p.L;
    const int r = n;
    constexpr int PER = NP >= 8 ? 1 : 8 / NP;  // outputs per lane per block
    const int base = NP >= 16 ? (r >> 1) : (NP >= 8 ? r : r * PER);
    // pass 2: from the carry, with the output.  Every lane of the CTA runs the
    // same number of 8-step blocks (steps past the segment end, or past L, are
    // the identity step with C = 0), so the warp-wide shuffles stay converged.
    const int nblk = p.seg_len / 8;
    for (int jb = 0; jb < nblk; ++jb) {
        const int t = s * p.seg_len + 8 * jb;
        float a[8], b[8], c[8], v[8];
        if (nv && t < t1) {
            load8<float>(ra, t, t1, vec, a, 1.0f);
            load8<float>(rb, t, t1, vec, b, 0.0f);
            load8<T>(rc, t, t1, vec, c, 0.0f);
        } else {
#pragma unroll
            for (int j = 0; j < 8; ++j) a[j] = 1.0f, b[j] = 0.0f, c[j] = 0.0f;
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            h = fmaf(a[j], h, b[j]);
            v[j] = c[j] * h;
        }
        reduce8<NP>(v, r);
        if (t < t1 && (NP < 16 || (r & 1) == 0)) {
#pragma unroll
            for (int j = 0; j < PER; ++j)
                if (t + base + j < t1) yr[t + base + j] = v[j];
        }
    }
}

template <typename T>
const void* only_fn(int np) {
    switch (np) {
    case 1: return reinterpret_cast<const void*>(&scan_only_kernel<T, 1>);
    case 2: return reinterpret_cast<const void*>(&scan_only_kernel<T, 2>);
    case 4: return reinterpret_cast<const void*>(&scan_only_kernel<T, 4>);
    case 8: return reinterpret_cast<const void*>(&scan_only_kernel<T, 8>);
    default: return reinterpret_cast<const void*>(&scan_only_kernel<T, 16>);
    }
}

int only_segments(int np) { return np >= 4 ? 64 : 256 / np; }

}  // namespace

vmb_status launch_discretise(const DiscArgs& a, bool mean, cudaStream_t stream) {
    DiscParams p{};
    p.u = a.u;
    p.dl = a.delta;
    p.A = a.A;
    p.Bs = a.Bs;
    p.bias = a.bias;
    p.dA = a.dA;
    p.dBu = a.dBu;
    p.K = a.K;
    p.D = a.D;
    p.N = a.N;
    p.L = a.L;
    p.softplus_on = (a.flags & VMB_FLAG_SOFTPLUS) ? 1 : 0;
    const bool zoh = (a.flags & VMB_FLAG_B_ZOH) != 0;
    const bool bf = a.dtype == VMB_BF16;
    const void* fn;
    long long grid;
    if (mean) {
        p.nlb = (a.L + kMeanSteps - 1) / kMeanSteps;
        grid = (long long)a.B * a.K * p.nlb;
        fn = bf ? (zoh ? reinterpret_cast<const void*>(&discretise_mean_kernel<__nv_bfloat16, true>)
                       : reinterpret_cast<const void*>(&discretise_mean_kernel<__nv_bfloat16, false>))
                : (zoh ? reinterpret_cast<const void*>(&discretise_mean_kernel<float, true>)
                       : reinterpret_cast<const void*>(&discretise_mean_kernel<float, false>));
    } else {
        p.nlb = (a.L + kDiscThreads - 1) / kDiscThreads;
        grid = (long long)a.B * a.K * a.D * p.nlb;
        fn = bf ? (zoh ? reinterpret_cast<const void*>(&discretise_kernel<__nv_bfloat16, true>)
                       : reinterpret_cast<const void*>(&discretise_kernel<__nv_bfloat16, false>))
                : (zoh ? reinterpret_cast<const void*>(&discretise_kernel<float, true>)
                       : reinterpret_cast<const void*>(&discretise_kernel<float, false>));
    }
    if (grid > INT32_MAX) return VMB_ERR_UNSUPPORTED;
    void* args[] = {&p};
    return launch_kernel(fn, dim3((unsigned)grid), dim3(kDiscThreads), 0, args, stream) == cudaSuccess ? VMB_OK
                                                                                                          : VMB_ERR_CUDA;
}

vmb_status launch_scan_only(const OnlyArgs& a, cudaStream_t stream) {
    OnlyParams p{};
    p.dA = a.dA;
    p.dBu = a.dBu;
    p.Cs = a.Cs;
    p.y = a.y;
    p.channels = (long long)a.B * a.K * a.Dm;
    p.Dm = a.Dm;
    p.N = a.N;
    p.L = a.L;
    const int np = a.N <= 1 ? 1 : a.N <= 2 ? 2 : a.N <= 4 ? 4 : a.N <= 8 ? 8 : 16;
    const int S = only_segments(np);
    p.seg_len = (int)(((long long)a.L + S - 1) / S);
    p.seg_len = (p.seg_len + 7) / 8 * 8;
    const size_t es = a.dtype == VMB_BF16 ? 2 : 4;
    const auto al = [](const void* q, size_t b) { return (reinterpret_cast<uintptr_t>(q) % b) == 0; };
    // every 8-step block starts 32 bytes into an fp32 row (16 into a bf16 one)
    p.vec = (a.L % 8 == 0) && al(a.dA, 32) && al(a.dBu, 32) && al(a.Cs, 8 * es) ? 1 : 0;
    const int threads = S * np;
    const long long grid = p.channels;
    if (grid > INT32_MAX) return VMB_ERR_UNSUPPORTED;
    const void* fn = a.dtype == VMB_BF16 ? only_fn<__nv_bfloat16>(np) : only_fn<float>(np);
    void* args[] = {&p};
    return launch_kernel(fn, dim3((unsigned)grid), dim3(threads), 0, args, stream) == cudaSuccess ? VMB_OK
                                                                                                   : VMB_ERR_CUDA;
}

}  // namespace vmb
