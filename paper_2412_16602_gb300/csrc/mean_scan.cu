// mean_scan.cu - VMeanba channel-mean selective scan (Sec. 2.2, Eq. 9) for sm_103a.
//
// y = T^-1(Mamba(T(Abar, Bbar u, C))): T averages the discretised scan inputs
// over the D channels of one (batch, direction), the recurrence runs once on
// the averages, and T^-1 broadcasts its output back to every channel.
//
// One CTA owns one (batch, direction) and one chunk of TC steps.
//   A. Channel reduction, fused into the load: the chunk's u and delta are
//      streamed through shared memory in sub-tiles of kDS channels (cp.async,
//      double buffered); each element gets its softplus once; thread (t, g, s)
//      accumulates sum_d 2^(delta_{d,t} A_{c,n} log2 e) for its NG states n
//      over its share s of the channels, and sum_d delta_{d,t} u_{d,t}.  Abar
//      is averaged after the exponential (Eq. 9 averages Abar itself).
//   B. The one-channel recurrence on the averages: micro-chunks of 8 steps per
//      (state, micro-chunk) thread, a serial combine over the micro-chunks, a
//      decoupled look-back over the preceding chunks of the same (batch,
//      direction) for the carry-in state, then the exact states and
//      ybar_t = sum_n C_{t,n} h_{t,n}.
//   C. Broadcast + skip: y[d, t] = ybar_t + Dskip_c u[d, t] for every channel,
//      written with 16-byte stores (u is read again; it is still in L2).
// The recurrence and the C.h work run once per (b, k) instead of once per
// (b, k, d); the exponentials of Abar stay per (b, k, d, n) because the mean
// is taken after them.
#include <mutex>

#include "vmb_common.cuh"
#include "vmb_internal.h"

namespace vmb {
namespace {

constexpr int kThreads = 256;
constexpr int kDS = 32;     // channels per reduction sub-tile
constexpr int kMC = 8;      // steps per micro-chunk of the local scan

struct MeanParams {
    const void* u;
    const void* dl;
    const float* A;
    const void* Bs;
    const void* Cs;
    const float* Dskip;
    const float* bias;
    void* y;
    float* ybar;
    int K, D, N, L;
    int softplus_on, skip_mean;
    int n_chunks, chunk_len, n_seq;
    int vec;
    int suppress;
    WsHeader* hdr;
    unsigned* flags;
    float* aggP;
    float* aggH;
    float* incH;
};

__host__ __device__ constexpr size_t a16(size_t v) { return (v + 15) / 16 * 16; }

template <typename T, int NP, int TC>
struct MLayout {
    static constexpr int NG = NP < 4 ? NP : 4;
    static constexpr int G = NP / NG;
    static constexpr int ITEMS = TC * G;             // (t, g) reduction items
    static constexpr int S = kThreads / ITEMS;       // channel splits
    static constexpr int TCF = TC + 1;
    static constexpr int RAW = 2 * kDS * TC;         // u + delta sub-tile
    static constexpr size_t raw_bytes = a16((size_t)2 * RAW * sizeof(T));
    static constexpr size_t dlf_off = raw_bytes;
    static constexpr size_t uf_off = dlf_off + (size_t)kDS * TCF * 4;
    static constexpr size_t a2_off = a16(uf_off + (size_t)kDS * TCF * 4);
    static constexpr size_t ar_off = a2_off + (size_t)kDS * NP * 4;
    static constexpr size_t dsk_off = ar_off + (size_t)kDS * NP * 4;
    static constexpr size_t bias_off = dsk_off + (size_t)kDS * 4;
    static constexpr size_t red_off = a16(bias_off + (size_t)kDS * 4);     // [S][TC][NP] x 2
    static constexpr size_t redu_off = red_off + (size_t)2 * S * TC * NP * 4;  // [S][TC] x 2
    static constexpr size_t abar_off = a16(redu_off + (size_t)2 * S * TC * 4);
    static constexpr size_t bubar_off = abar_off + (size_t)TC * NP * 4;
    static constexpr size_t bf_off = bubar_off + (size_t)TC * NP * 4;
    static constexpr size_t cf_off = bf_off + (size_t)TC * NP * 4;
    static constexpr size_t mc_off = cf_off + (size_t)TC * NP * 4;          // [4][TC/kMC][NP]
    static constexpr size_t ybar_off = mc_off + (size_t)4 * (TC / kMC) * NP * 4;
    static constexpr size_t dsu_off = ybar_off + (size_t)TC * 4;
    static constexpr size_t hin_off = dsu_off + (size_t)TC * 4;
    static constexpr size_t bytes = hin_off + (size_t)NP * 4;
    static_assert(S >= 1 && kThreads % ITEMS == 0, "items must divide the block");
    static_assert(bytes <= 100 * 1024, "mean-scan tile must leave room for two CTAs per SM");
    static_assert(TC % kMC == 0 && NP * (TC / kMC) <= kThreads, "local scan mapping");
};

template <typename T, int NP, int TC, bool ZOH>
__global__ void __launch_bounds__(kThreads) mean_scan_kernel(const MeanParams p) {
    using LY = MLayout<T, NP, TC>;
    constexpr int NG = LY::NG, G = LY::G, S = LY::S, TCF = LY::TCF, RAW = LY::RAW;
    constexpr int NMC = TC / kMC;
    extern __shared__ __align__(16) unsigned char smem[];
    T* raw = reinterpret_cast<T*>(smem);
    float* dlf = reinterpret_cast<float*>(smem + LY::dlf_off);
    float* uf = reinterpret_cast<float*>(smem + LY::uf_off);
    float* s_a2 = reinterpret_cast<float*>(smem + LY::a2_off);
    float* s_ar = reinterpret_cast<float*>(smem + LY::ar_off);
    float* s_dsk = reinterpret_cast<float*>(smem + LY::dsk_off);
    float* s_bias = reinterpret_cast<float*>(smem + LY::bias_off);
    float* red = reinterpret_cast<float*>(smem + LY::red_off);
    float* redu = reinterpret_cast<float*>(smem + LY::redu_off);
    float* abar = reinterpret_cast<float*>(smem + LY::abar_off);
    float* bubar = reinterpret_cast<float*>(smem + LY::bubar_off);
    float* bfm = reinterpret_cast<float*>(smem + LY::bf_off);
    float* cfm = reinterpret_cast<float*>(smem + LY::cf_off);
    float* mcP = reinterpret_cast<float*>(smem + LY::mc_off);
    float* mcH = mcP + NMC * NP;
    float* exP = mcH + NMC * NP;
    float* exH = exP + NMC * NP;
    float* s_ybar = reinterpret_cast<float*>(smem + LY::ybar_off);
    float* s_dsu = reinterpret_cast<float*>(smem + LY::dsu_off);
    float* s_hin = reinterpret_cast<float*>(smem + LY::hin_off);
    __shared__ unsigned s_misc[2];

    const int tid = threadIdx.x;
    const bool chunked = p.n_chunks > 1;
    int seq, chunk;
    unsigned gen = 0;
    if (chunked) {
        if (tid == 0) {
            s_misc[0] = atomicAdd(&p.hdr->ticket, 1u);
            s_misc[1] = ld_relaxed(&p.hdr->gen);
        }
        __syncthreads();
        const unsigned t = s_misc[0];
        gen = s_misc[1];
        if (t >= (unsigned)(p.n_seq * p.n_chunks)) {  // workspace was not zero-filled
            if (tid == 0) {
                atomicOr(&p.hdr->err, kErrBounds);
                finish_launch(p.hdr, (unsigned)(p.n_seq * p.n_chunks));
            }
            return;
        }
        chunk = (int)(t / (unsigned)p.n_seq);
        seq = (int)(t % (unsigned)p.n_seq);
    } else {
        seq = blockIdx.x;
        chunk = 0;
    }
    const int k = seq % p.K;
    const int D = p.D, L = p.L, N = p.N;
    const int l0 = chunk * p.chunk_len;
    const int nvalid = min(TC, L - l0);
    const size_t urow0 = (size_t)seq * D;   // first row of u/delta/y for (b, k)
    const size_t bcrow0 = (size_t)seq * N;  // first row of Bs/Cs
    const T* u = static_cast<const T*>(p.u);
    const T* dlr = static_cast<const T*>(p.dl);

    // B and C of the chunk, transposed to [t][n]
    for (int i = tid; i < NP * TC; i += kThreads) {
        const int n = i / TC, t = i % TC;
        const bool ok = n < N && t < nvalid;
        const size_t gi = (bcrow0 + n) * (size_t)L + l0 + t;
        bfm[t * NP + n] = ok ? io<T>::ld(static_cast<const T*>(p.Bs) + gi) : 0.0f;
        cfm[t * NP + n] = ok ? io<T>::ld(static_cast<const T*>(p.Cs) + gi) : 0.0f;
    }

    // ---------------------------------------------------------------- phase A
    const int item = tid % LY::ITEMS;
    const int sidx = tid / LY::ITEMS;
    const int rt = item % TC;  // step of this reduction item
    const int rg = item / TC;  // state group of this reduction item
    float acc[NG], accb[NG];
#pragma unroll
    for (int i = 0; i < NG; ++i) {
        acc[i] = 0.0f;
        accb[i] = 0.0f;
    }
    float sdu = 0.0f, sdsu = 0.0f;

    const int nsub = (D + kDS - 1) / kDS;
    auto load_sub = [&](int st, T* dst) {
        const int r0 = st * kDS;
        const int nr = min(kDS, D - r0);
        if (p.vec) {
            constexpr int VE = 16 / sizeof(T), CPR = TC / VE;
            for (int i = tid; i < 2 * kDS * CPR; i += kThreads) {
                const int which = i / (kDS * CPR);
                const int j = i % (kDS * CPR);
                const int r = j / CPR, ch = j % CPR;
                const T* base = which ? dlr : u;
                const bool ok = r < nr && ch * VE < nvalid;
                const T* src = ok ? base + (urow0 + r0 + r) * (size_t)L + l0 + ch * VE : base;
                cp_async16(dst + which * kDS * TC + r * TC + ch * VE, src, ok ? 16 : 0);
            }
        } else {
            for (int i = tid; i < 2 * kDS * TC; i += kThreads) {
                const int which = i / (kDS * TC);
                const int j = i % (kDS * TC);
                const int r = j / TC, t = j % TC;
                const T* base = which ? dlr : u;
                T v = T(0.0f);
                if (r < nr && t < nvalid) v = base[(urow0 + r0 + r) * (size_t)L + l0 + t];
                dst[i] = v;
            }
        }
    };

    load_sub(0, raw);
    cp_async_commit();
    for (int st = 0; st < nsub; ++st) {
        if (st + 1 < nsub) load_sub(st + 1, raw + ((st + 1) & 1) * RAW);
        cp_async_commit();
        cp_async_wait<1>();
        const int r0 = st * kDS;
        const int nr = min(kDS, D - r0);
        // per-channel tables of the sub-tile
        for (int i = tid; i < kDS * NP; i += kThreads) {
            const int r = i / NP, n = i % NP;
            const float a = (r < nr && n < N) ? p.A[((size_t)k * D + r0 + r) * N + n] : 0.0f;
            s_a2[i] = a * kLog2e;
            s_ar[i] = a;
        }
        for (int i = tid; i < kDS; i += kThreads) {
            s_bias[i] = i < nr ? p.bias[(size_t)k * D + r0 + i] : 0.0f;
            s_dsk[i] = i < nr ? p.Dskip[(size_t)k * D + r0 + i] : 0.0f;
        }
        __syncthreads();
        // conversion: softplus once per element
        {
            const T* ru = raw + (st & 1) * RAW;
            const T* rd = ru + kDS * TC;
            for (int i = tid; i < kDS * TC; i += kThreads) {
                const int r = i / TC, t = i % TC;
                const bool ok = r < nr && t < nvalid;
                const float v = io<T>::cvt(rd[i]) + s_bias[r];
                const float dv = p.softplus_on ? softplus(v) : v;
                dlf[r * TCF + t] = ok ? dv : 0.0f;
                uf[r * TCF + t] = ok ? io<T>::cvt(ru[i]) : 0.0f;
            }
        }
        __syncthreads();
        // reduction over this thread's channels of the sub-tile
        for (int r = sidx; r < nr; r += S) {
            const float dv = dlf[r * TCF + rt];
            const float uv = uf[r * TCF + rt];
            const float* a2 = s_a2 + r * NP + rg * NG;
            if constexpr (ZOH) {
                const float* ar = s_ar + r * NP + rg * NG;
#pragma unroll
                for (int i = 0; i < NG; ++i) {
                    const float em1 = expm1f(dv * ar[i]);
                    acc[i] += 1.0f + em1;
                    accb[i] = fmaf(ar[i] != 0.0f ? em1 / ar[i] : dv, uv, accb[i]);
                }
            } else if constexpr (NG % 2 == 0) {
#pragma unroll
                for (int i = 0; i < NG; i += 2) {
                    const float2 x = __fmul2_rn(make_float2(dv, dv), make_float2(a2[i], a2[i + 1]));
                    const float2 e = make_float2(ex2(x.x), ex2(x.y));
                    const float2 s2 = __fadd2_rn(make_float2(acc[i], acc[i + 1]), e);
                    acc[i] = s2.x;
                    acc[i + 1] = s2.y;
                }
            } else {
#pragma unroll
                for (int i = 0; i < NG; ++i) acc[i] += ex2(dv * a2[i]);
            }
            if (rg == 0) sdu = fmaf(dv, uv, sdu);
            if (p.skip_mean && rg == G - 1) sdsu = fmaf(s_dsk[r], uv, sdsu);
        }
    }
    cp_async_wait<0>();

    // ---------------------------------------------------------------- phase B
    // partial sums of the S channel splits -> averages
#pragma unroll
    for (int i = 0; i < NG; ++i) {
        red[(sidx * TC + rt) * NP + rg * NG + i] = acc[i];
        red[S * TC * NP + (sidx * TC + rt) * NP + rg * NG + i] = accb[i];
    }
    if (rg == 0) redu[sidx * TC + rt] = sdu;
    if (rg == G - 1) redu[S * TC + sidx * TC + rt] = sdsu;
    __syncthreads();
    const float invD = 1.0f / (float)D;
    for (int i = tid; i < TC * NP; i += kThreads) {
        const int t = i / NP;
        float sa = 0.0f, sb = 0.0f, su = 0.0f;
#pragma unroll
        for (int s = 0; s < S; ++s) {
            sa += red[s * TC * NP + i];
            sb += red[S * TC * NP + s * TC * NP + i];
            su += redu[s * TC + t];
        }
        abar[i] = sa * invD;
        bubar[i] = bfm[i] * (ZOH ? sb : su) * invD;
    }
    for (int t = tid; t < TC; t += kThreads) {
        float sd = 0.0f;
#pragma unroll
        for (int s = 0; s < S; ++s) sd += redu[S * TC + s * TC + t];
        s_dsu[t] = sd * invD;
    }
    __syncthreads();
    // local scan of each micro-chunk (from h = 0)
    if (tid < NP * NMC) {
        const int n = tid % NP, m = tid / NP;
        float P = 1.0f, H = 0.0f;
#pragma unroll
        for (int j = 0; j < kMC; ++j) {
            const int t = m * kMC + j;
            const float a = abar[t * NP + n];
            H = fmaf(a, H, bubar[t * NP + n]);
            P *= a;
        }
        mcP[m * NP + n] = P;
        mcH[m * NP + n] = H;
    }
    __syncthreads();
    // serial combine over micro-chunks: exclusive prefixes and the chunk aggregate
    if (tid < NP) {
        const int n = tid;
        float P = 1.0f, H = 0.0f;
        for (int m = 0; m < NMC; ++m) {
            exP[m * NP + n] = P;
            exH[m * NP + n] = H;
            const float mp = mcP[m * NP + n];
            H = fmaf(mp, H, mcH[m * NP + n]);
            P *= mp;
        }
        float hin = 0.0f;
        if (chunked) {
            const size_t slot = (size_t)seq * p.n_chunks + chunk;
            if (chunk == 0) {
                p.incH[slot * NP + n] = H;
            } else {
                p.aggP[slot * NP + n] = P;
                p.aggH[slot * NP + n] = H;
            }
            __threadfence();
        }
        s_hin[n] = H;  // temporarily: the chunk's local end state
        mcP[n] = P;    // temporarily: the chunk's product (mcP is no longer needed)
        (void)hin;
    }
    __syncthreads();
    if (chunked) {
        const size_t slot = (size_t)seq * p.n_chunks + chunk;
        if (tid == 0 && !(p.suppress && chunk == 0))
            st_release(&p.flags[slot], flag_word(gen, chunk == 0 ? kFlagInclusive : kFlagAggregate));
        float RH = 0.0f;
        if (chunk > 0) {
            // Decoupled look-back with a left fold after the inclusive state found
            // (bit-identical carry whichever predecessor the walk stops at).
            int found = -1;
            for (int j = chunk - 1; j >= 0; --j) {
                const size_t sj = (size_t)seq * p.n_chunks + j;
                if (tid == 0) s_misc[0] = wait_flag(&p.flags[sj], gen, p.hdr, (unsigned)seq, (unsigned)j);
                __syncthreads();
                const unsigned kind = s_misc[0];
                __syncthreads();
                if (kind == kFlagInclusive) {
                    found = j;
                    break;
                }
                if (kind != kFlagAggregate) break;
            }
            if (found >= 0 && tid < NP) {
                RH = ld_cg(&p.incH[((size_t)seq * p.n_chunks + found) * NP + tid]);
                for (int m = found + 1; m < chunk; ++m) {
                    const size_t sm = (size_t)seq * p.n_chunks + m;
                    RH = fmaf(ld_cg(&p.aggP[sm * NP + tid]), RH, ld_cg(&p.aggH[sm * NP + tid]));
                }
            }
            if (tid < NP) {
                p.incH[slot * NP + tid] = fmaf(mcP[tid], RH, s_hin[tid]);
                __threadfence();
            }
            __syncthreads();
            if (tid == 0) st_release(&p.flags[slot], flag_word(gen, kFlagInclusive));
        }
        __syncthreads();
        if (tid < NP) s_hin[tid] = RH;  // carry-in state of this chunk
    } else {
        if (tid < NP) s_hin[tid] = 0.0f;
    }
    __syncthreads();
    // exact states of each micro-chunk and C . h  (written into abar as scratch)
    if (tid < NP * NMC) {
        const int n = tid % NP, m = tid / NP;
        float h = fmaf(exP[m * NP + n], s_hin[n], exH[m * NP + n]);
#pragma unroll
        for (int j = 0; j < kMC; ++j) {
            const int t = m * kMC + j;
            h = fmaf(abar[t * NP + n], h, bubar[t * NP + n]);
            abar[t * NP + n] = cfm[t * NP + n] * h;
        }
    }
    __syncthreads();
    for (int t = tid; t < TC; t += kThreads) {
        float s = 0.0f;
#pragma unroll
        for (int n = 0; n < NP; ++n) s += abar[t * NP + n];
        s_ybar[t] = s;
        if (p.ybar && t < nvalid) p.ybar[(size_t)seq * L + l0 + t] = s;
    }
    __syncthreads();

    // ---------------------------------------------------------------- phase C
    T* y = static_cast<T*>(p.y);
    if (p.vec) {
        constexpr int VE = 16 / sizeof(T), CPR = TC / VE;
        for (int i = tid; i < D * CPR; i += kThreads) {
            const int r = i / CPR, ch = i % CPR;
            if (ch * VE >= nvalid) continue;
            const size_t gi = (urow0 + r) * (size_t)L + l0 + ch * VE;
            const float dsk = p.Dskip[(size_t)k * D + r];
            union { uint4 v; T e[VE]; } in, out;
            in.v = *reinterpret_cast<const uint4*>(u + gi);
#pragma unroll
            for (int e = 0; e < VE; ++e) {
                const int t = ch * VE + e;
                const float skip = p.skip_mean ? s_dsu[t] : dsk * io<T>::cvt(in.e[e]);
                out.e[e] = io<T>::to(s_ybar[t] + skip);
            }
            *reinterpret_cast<uint4*>(y + gi) = out.v;
        }
    } else {
        for (int i = tid; i < D * TC; i += kThreads) {
            const int r = i / TC, t = i % TC;
            if (t >= nvalid) continue;
            const size_t gi = (urow0 + r) * (size_t)L + l0 + t;
            const float skip = p.skip_mean ? s_dsu[t] : p.Dskip[(size_t)k * D + r] * io<T>::ld(u + gi);
            y[gi] = io<T>::to(s_ybar[t] + skip);
        }
    }

    if (chunked) {
        __syncthreads();
        if (tid == 0) finish_launch(p.hdr, (unsigned)(p.n_seq * p.n_chunks));
    }
}

// ------------------------------------------------------------------ host side

struct KInfo {
    const void* fn;
    size_t smem;
};

template <typename T, int NP, int TC, bool ZOH>
KInfo minfo() {
    using LY = MLayout<T, NP, TC>;
    const void* fn = reinterpret_cast<const void*>(&mean_scan_kernel<T, NP, TC, ZOH>);
    static std::once_flag once;
    static cudaError_t err = cudaSuccess;
    std::call_once(once, [&] {
        err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)LY::bytes);
    });
    if (err != cudaSuccess) return {nullptr, 0};
    return {fn, LY::bytes};
}

template <typename T, int NP, bool ZOH>
KInfo pick_tc(int tc) {
    switch (tc) {
    case 16: return minfo<T, NP, 16, ZOH>();
    case 32: return minfo<T, NP, 32, ZOH>();
    default: return minfo<T, NP, 64, ZOH>();
    }
}

template <typename T, bool ZOH>
KInfo pick_np(int np, int tc) {
    switch (np) {
    case 1: return pick_tc<T, 1, ZOH>(tc);
    case 2: return pick_tc<T, 2, ZOH>(tc);
    case 4: return pick_tc<T, 4, ZOH>(tc);
    case 8: return pick_tc<T, 8, ZOH>(tc);
    default: return pick_tc<T, 16, ZOH>(tc);
    }
}

KInfo mpick(vmb_dtype dt, int np, int tc, bool zoh) {
    if (dt == VMB_BF16) return zoh ? pick_np<__nv_bfloat16, true>(np, tc) : pick_np<__nv_bfloat16, false>(np, tc);
    return zoh ? pick_np<float, true>(np, tc) : pick_np<float, false>(np, tc);
}

}  // namespace

vmb_status plan_mean(const ScanArgs& a, ScanPlan* plan) {
    if (a.N < 1 || a.N > 16) return VMB_ERR_UNSUPPORTED;
    int np = 1;
    while (np < a.N) np <<= 1;
    const bool zoh = (a.flags & VMB_FLAG_B_ZOH) != 0;
    // Largest chunk length whose grid still fills the GPU (one CTA per (b, k, chunk)).
    const long long seqs = (long long)a.B * a.K;
    int tc = 16;
    for (int cand : {64, 32, 16}) {
        KInfo ki = mpick(a.dtype, np, cand, zoh);
        if (!ki.fn) return VMB_ERR_CUDA;
        int per_sm = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, ki.fn, kThreads, ki.smem) != cudaSuccess)
            return VMB_ERR_CUDA;
        const long long resident = (long long)(per_sm < 1 ? 1 : per_sm) * device_sm_count();
        if (seqs * ((a.L + cand - 1) / cand) >= resident || cand == 16) {
            tc = cand;
            break;
        }
    }
    ScanPlan p{};
    p.np = np;
    p.tile_rows = 0;
    p.tiles_per_bk = 1;
    p.n_seq = (int)seqs;
    p.chunk_len = tc;
    p.n_chunks = (a.L + tc - 1) / tc;
    p.state_floats = (size_t)np;
    p.ws_bytes = ws_layout(p).total;
    *plan = p;
    return VMB_OK;
}

vmb_status launch_mean(const ScanArgs& a, const ScanPlan& plan, cudaStream_t stream) {
    KInfo ki = mpick(a.dtype, plan.np, plan.chunk_len, (a.flags & VMB_FLAG_B_ZOH) != 0);
    if (!ki.fn) return VMB_ERR_CUDA;
    const size_t es = a.dtype == VMB_BF16 ? 2 : 4;
    MeanParams p{};
    p.u = a.u;
    p.dl = a.delta;
    p.A = a.A;
    p.Bs = a.Bs;
    p.Cs = a.Cs;
    p.Dskip = a.Dskip;
    p.bias = a.bias;
    p.y = a.y;
    p.ybar = a.ybar;
    p.K = a.K;
    p.D = a.D;
    p.N = a.N;
    p.L = a.L;
    p.softplus_on = (a.flags & VMB_FLAG_SOFTPLUS) ? 1 : 0;
    p.skip_mean = (a.flags & VMB_FLAG_SKIP_MEAN) ? 1 : 0;
    p.n_chunks = plan.n_chunks;
    p.chunk_len = plan.chunk_len;
    p.n_seq = plan.n_seq;
    const auto al16 = [](const void* q) { return (reinterpret_cast<uintptr_t>(q) & 15u) == 0; };
    p.vec = ((size_t)a.L * es % 16 == 0) && al16(a.u) && al16(a.delta) && al16(a.y);
    p.suppress = (a.flags & VMB_FLAG_TEST_SUPPRESS_PUBLISH) ? 1 : 0;
    const WsLayout w = ws_layout(plan);
    unsigned char* ws = static_cast<unsigned char*>(a.ws);
    p.hdr = reinterpret_cast<WsHeader*>(ws);
    p.flags = reinterpret_cast<unsigned*>(ws + w.flags_off);
    p.aggP = reinterpret_cast<float*>(ws + w.aggP_off);
    p.aggH = reinterpret_cast<float*>(ws + w.aggH_off);
    p.incH = reinterpret_cast<float*>(ws + w.incH_off);
    const unsigned grid = (unsigned)(plan.n_seq * plan.n_chunks);
    void* args[] = {&p};
    cudaError_t e = cudaLaunchKernel(ki.fn, dim3(grid), dim3(kThreads), args, ki.smem, stream);
    return e == cudaSuccess ? VMB_OK : VMB_ERR_CUDA;
}

}  // namespace vmb
