// full_scan.cu - full-channel selective scan (App. A, Eqs. 3, 4, 6) for sm_103a.
//
// One CTA owns a tile of DT = 256/G channels of one (batch, direction) and one
// chunk of the sequence.  Each thread owns one channel and NG = NP/G of its
// NP states (G threads per channel, adjacent lanes).  The CTA streams its
// chunk through shared memory in stages of kTS steps (cp.async, double
// buffered); a conversion pass turns each stage into fp32, applies the
// softplus of Eq. 6 once per element, and transposes B and C to [t][n] so a
// thread reads its states as one vector.  Discretisation (Eq. 4) happens in
// registers: Abar = 2^(delta * A log2 e) on the MUFU pipe, Bbar u = delta u B.
// The per-channel output y = sum_n C_n h_n + D u is reduced across the G lanes
// with a transposed butterfly (lane g ends with step t0+g), staged in shared
// memory and written back with 16-byte stores.
//
// Long sequences with few channels are cut into L-chunks that run in
// parallel.  Chunks after the first run twice: a first pass computes the
// chunk's aggregate (P = prod Abar, H = end state from h = 0) and publishes
// it; a decoupled look-back over the predecessors' aggregates and inclusive
// end states gives the carry-in state; the second pass recomputes the chunk
// from that state and writes y.  The first chunk of a sequence runs once and
// publishes its end state.  Chunk order is fixed by a ticket counter so that a
// CTA only ever waits on CTAs that started before it; every wait is bounded.
#include <mutex>
#include <type_traits>

#include "vmb_common.cuh"
#include "vmb_internal.h"

namespace vmb {
namespace {

constexpr int kStages = 2;

struct FullParams {
    const void* u;
    const void* dl;
    const float* A;
    const void* Bs;
    const void* Cs;
    const float* Dskip;
    const float* bias;
    void* y;
    int K, D, N, L;
    int softplus_on;
    int tiles_per_bk, n_tiles, n_chunks, chunk_len;
    int vec;       // rows are 16-byte aligned: cp.async 16-byte path
    int suppress;  // test hook: chunk 0 does not publish
    WsHeader* hdr;
    unsigned* flags;
    float* aggP;
    float* aggH;
    float* incH;
};

__host__ __device__ constexpr size_t a16(size_t v) { return (v + 15) / 16 * 16; }

// Tile shape per state split G: 64 channels x 32-step stages when four lanes
// share a channel (N = 16), 128 channels x 16-step stages otherwise, so that
// a CTA's shared memory stays near 60 KB and three or more CTAs fit per SM.
template <typename T, int NP, int G>
struct Layout {
    static constexpr int DT = G == 4 ? 64 : 128;
    static constexpr int THREADS = DT * G;
    static constexpr int TS = G == 4 ? 32 : 16;
    static constexpr int TSF = TS + 1;
    static constexpr int RAW = (2 * DT + 2 * NP) * TS;  // elements per raw stage
    static constexpr size_t raw_bytes = a16((size_t)kStages * RAW * sizeof(T));
    static constexpr size_t uf_off = raw_bytes;
    static constexpr size_t df_off = uf_off + (size_t)DT * TSF * 4;
    static constexpr size_t bf_off = a16(df_off + (size_t)DT * TSF * 4);
    static constexpr size_t cf_off = bf_off + (size_t)TS * NP * 4;
    static constexpr size_t ys_off = a16(cf_off + (size_t)TS * NP * 4);
    static constexpr size_t bias_off = a16(ys_off + (size_t)DT * TS * sizeof(T));
    static constexpr size_t bytes = bias_off + (size_t)DT * 4;
    static_assert(bytes <= 100 * 1024, "full-scan tile must leave room for two CTAs per SM");
};

// Sum of yp[j] over the G lanes of one channel; lane g returns the sum for j = g.
template <int G>
__device__ __forceinline__ float reduce_lanes(const float (&yp)[G], int g) {
    if constexpr (G == 1) {
        return yp[0];
    } else if constexpr (G == 2) {
        float keep = g ? yp[1] : yp[0];
        float send = g ? yp[0] : yp[1];
        return keep + __shfl_xor_sync(0xffffffffu, send, 1);
    } else {
        static_assert(G == 4, "G in {1, 2, 4}");
        const bool hi = g & 2;
        float k0 = hi ? yp[2] : yp[0], k1 = hi ? yp[3] : yp[1];
        float s0 = hi ? yp[0] : yp[2], s1 = hi ? yp[1] : yp[3];
        k0 += __shfl_xor_sync(0xffffffffu, s0, 2);
        k1 += __shfl_xor_sync(0xffffffffu, s1, 2);
        const bool odd = g & 1;
        float kk = odd ? k1 : k0, ss = odd ? k0 : k1;
        return kk + __shfl_xor_sync(0xffffffffu, ss, 1);
    }
}

template <typename T, int NP, int G, bool WITH_C>
__device__ __forceinline__ void load_stage(const FullParams& p, T* dst, size_t row0, size_t bcrow0,
                                           int nrows, int l0) {
    using LY = Layout<T, NP, G>;
    constexpr int DT = LY::DT;
    constexpr int kTS = LY::TS;
    constexpr int kThreads = LY::THREADS;
    constexpr int VE = 16 / sizeof(T);  // elements per 16-byte chunk
    constexpr int CPR = kTS / VE;       // chunks per stage row
    const T* u = static_cast<const T*>(p.u);
    const T* dl = static_cast<const T*>(p.dl);
    const T* Bs = static_cast<const T*>(p.Bs);
    const T* Cs = static_cast<const T*>(p.Cs);
    const int L = p.L;
    if (p.vec) {
        constexpr int nU = DT * CPR, nB = NP * CPR;
        constexpr int total = 2 * nU + (WITH_C ? 2 : 1) * nB;
        for (int i = threadIdx.x; i < total; i += kThreads) {
            const T* src;
            T* d;
            bool ok;
            int r, ch;
            if (i < 2 * nU) {
                const int j = i < nU ? i : i - nU;
                r = j / CPR;
                ch = j % CPR;
                const T* base = i < nU ? u : dl;
                ok = r < nrows && l0 + ch * VE < L;
                src = ok ? base + ((row0 + r) * (size_t)L + l0 + ch * VE) : base;
                d = dst + (i < nU ? 0 : DT * kTS) + r * kTS + ch * VE;
            } else {
                const int i2 = i - 2 * nU;
                const int j = i2 < nB ? i2 : i2 - nB;
                r = j / CPR;
                ch = j % CPR;
                const T* base = i2 < nB ? Bs : Cs;
                ok = r < p.N && l0 + ch * VE < L;
                src = ok ? base + ((bcrow0 + r) * (size_t)L + l0 + ch * VE) : base;
                d = dst + 2 * DT * kTS + (i2 < nB ? 0 : NP * kTS) + r * kTS + ch * VE;
            }
            cp_async16(d, src, ok ? 16 : 0);
        }
    } else {
        constexpr int nU = DT * kTS, nB = NP * kTS;
        constexpr int total = 2 * nU + (WITH_C ? 2 : 1) * nB;
        for (int i = threadIdx.x; i < total; i += kThreads) {
            T v = T(0.0f);
            if (i < 2 * nU) {
                const int j = i < nU ? i : i - nU;
                const int r = j / kTS, t = j % kTS;
                const T* base = i < nU ? u : dl;
                if (r < nrows && l0 + t < L) v = base[(row0 + r) * (size_t)L + l0 + t];
            } else {
                const int i2 = i - 2 * nU;
                const int j = i2 < nB ? i2 : i2 - nB;
                const int r = j / kTS, t = j % kTS;
                const T* base = i2 < nB ? Bs : Cs;
                if (r < p.N && l0 + t < L) v = base[(bcrow0 + r) * (size_t)L + l0 + t];
            }
            dst[i] = v;
        }
    }
}

template <typename T, int NP, int G, bool ZOH>
__global__ void __launch_bounds__(Layout<T, NP, G>::THREADS) full_scan_kernel(const FullParams p) {
    using LY = Layout<T, NP, G>;
    constexpr int kThreads = LY::THREADS;
    constexpr int kTS = LY::TS;
    constexpr int NG = NP / G;
    constexpr int DT = LY::DT;
    constexpr int TSF = LY::TSF;
    constexpr int RAW = LY::RAW;
    extern __shared__ __align__(16) unsigned char smem[];
    T* raw = reinterpret_cast<T*>(smem);
    float* uf = reinterpret_cast<float*>(smem + LY::uf_off);
    float* df = reinterpret_cast<float*>(smem + LY::df_off);
    float* bfm = reinterpret_cast<float*>(smem + LY::bf_off);
    float* cfm = reinterpret_cast<float*>(smem + LY::cf_off);
    T* ys = reinterpret_cast<T*>(smem + LY::ys_off);
    float* s_bias = reinterpret_cast<float*>(smem + LY::bias_off);
    __shared__ unsigned s_misc[2];

    const int tid = threadIdx.x;
    int tile, chunk;
    unsigned gen = 0;
    const bool chunked = p.n_chunks > 1;
    if (chunked) {
        if (tid == 0) {
            s_misc[0] = atomicAdd(&p.hdr->ticket, 1u);
            s_misc[1] = ld_relaxed(&p.hdr->gen);
        }
        __syncthreads();
        const unsigned t = s_misc[0];
        gen = s_misc[1];
        if (t >= (unsigned)(p.n_tiles * p.n_chunks)) {  // workspace was not zero-filled
            if (tid == 0) {
                atomicOr(&p.hdr->err, kErrBounds);
                finish_launch(p.hdr, (unsigned)(p.n_tiles * p.n_chunks));
            }
            return;
        }
        chunk = (int)(t / (unsigned)p.n_tiles);
        tile = (int)(t % (unsigned)p.n_tiles);
    } else {
        tile = blockIdx.x;
        chunk = 0;
    }
    const int bk = tile / p.tiles_per_bk;
    const int d0 = (tile % p.tiles_per_bk) * DT;
    const int k = bk % p.K;
    const int c = tid / G, g = tid % G;
    const int d = d0 + c;
    const bool cval = d < p.D;
    const int nrows = min(DT, p.D - d0);
    const size_t row0 = (size_t)bk * p.D + d0;
    const size_t bcrow0 = (size_t)bk * p.N;

    for (int i = tid; i < DT; i += kThreads) s_bias[i] = i < nrows ? p.bias[(size_t)k * p.D + d0 + i] : 0.0f;

    float A2[NG], Ar[NG], h[NG], P[NG];
#pragma unroll
    for (int i = 0; i < NG; ++i) {
        const int n = g * NG + i;
        const float a = (cval && n < p.N) ? p.A[((size_t)k * p.D + d) * p.N + n] : 0.0f;
        A2[i] = a * kLog2e;
        Ar[i] = a;
        h[i] = 0.0f;
        P[i] = 1.0f;
    }
    const float dsk = cval ? p.Dskip[(size_t)k * p.D + d] : 0.0f;
    const int l_begin = chunk * p.chunk_len;
    const int l_end = min(p.L, l_begin + p.chunk_len);
    const int nst = (l_end - l_begin + kTS - 1) / kTS;
    __syncthreads();

    // One pass over the chunk.  PH2 = false: aggregate only (h from 0, P = prod Abar).
    // PH2 = true: recurrence from the carried-in h, output y.
    auto pass = [&](auto ph2_tag) {
        constexpr bool PH2 = decltype(ph2_tag)::value;
        load_stage<T, NP, G, PH2>(p, raw, row0, bcrow0, nrows, l_begin);
        cp_async_commit();
        for (int s = 0; s < nst; ++s) {
            const int l0 = l_begin + s * kTS;
            if (s + 1 < nst) load_stage<T, NP, G, PH2>(p, raw + ((s + 1) & 1) * RAW, row0, bcrow0, nrows, l0 + kTS);
            cp_async_commit();
            cp_async_wait<1>();
            __syncthreads();
            // ---- conversion: fp32, softplus(delta + bias), B/C transposed to [t][n]
            {
                const T* ru = raw + (s & 1) * RAW;
                const T* rd = ru + DT * kTS;
                const T* rb = rd + DT * kTS;
                const T* rc = rb + NP * kTS;
                const int nvalid = min(kTS, l_end - l0);
                for (int i = tid; i < DT * kTS; i += kThreads) {
                    const int r = i / kTS, t = i % kTS;
                    const bool ok = r < nrows && t < nvalid;
                    const float v = io<T>::cvt(rd[i]) + s_bias[r];
                    const float dv = p.softplus_on ? softplus(v) : v;
                    uf[r * TSF + t] = ok ? io<T>::cvt(ru[i]) : 0.0f;
                    df[r * TSF + t] = ok ? dv : 0.0f;
                }
                for (int i = tid; i < NP * kTS; i += kThreads) {
                    const int n = i / kTS, t = i % kTS;
                    const bool ok = n < p.N && t < nvalid;
                    bfm[t * NP + n] = ok ? io<T>::cvt(rb[i]) : 0.0f;
                    if constexpr (PH2) cfm[t * NP + n] = ok ? io<T>::cvt(rc[i]) : 0.0f;
                }
            }
            __syncthreads();
            // ---- recurrence over the stage
#pragma unroll 1
            for (int t0 = 0; t0 < kTS; t0 += G) {
                float yp[G];
#pragma unroll
                for (int j = 0; j < G; ++j) {
                    const int t = t0 + j;
                    const float dlt = df[c * TSF + t];
                    const float uu = uf[c * TSF + t];
                    const float du = dlt * uu;
                    float Bv[NG], Cv[NG];
#pragma unroll
                    for (int i = 0; i < NG; ++i) {
                        Bv[i] = bfm[t * NP + g * NG + i];
                        if constexpr (PH2) Cv[i] = cfm[t * NP + g * NG + i];
                    }
                    float ya = 0.0f, yb = 0.0f;
                    if constexpr (!ZOH && NG % 2 == 0) {
#pragma unroll
                        for (int i = 0; i < NG; i += 2) {
                            const float2 x = __fmul2_rn(make_float2(dlt, dlt), make_float2(A2[i], A2[i + 1]));
                            const float2 a = make_float2(ex2(x.x), ex2(x.y));
                            const float2 bb = __fmul2_rn(make_float2(du, du), make_float2(Bv[i], Bv[i + 1]));
                            const float2 hh = __ffma2_rn(a, make_float2(h[i], h[i + 1]), bb);
                            h[i] = hh.x;
                            h[i + 1] = hh.y;
                            if constexpr (PH2) {
                                const float2 acc = __ffma2_rn(make_float2(Cv[i], Cv[i + 1]), hh, make_float2(ya, yb));
                                ya = acc.x;
                                yb = acc.y;
                            } else {
                                const float2 pp = __fmul2_rn(make_float2(P[i], P[i + 1]), a);
                                P[i] = pp.x;
                                P[i + 1] = pp.y;
                            }
                        }
                    } else {
#pragma unroll
                        for (int i = 0; i < NG; ++i) {
                            float a, bb;
                            if constexpr (ZOH) {
                                const float em1 = expm1f(dlt * Ar[i]);
                                a = 1.0f + em1;
                                bb = (Ar[i] != 0.0f ? em1 / Ar[i] : dlt) * Bv[i] * uu;
                            } else {
                                a = ex2(dlt * A2[i]);
                                bb = du * Bv[i];
                            }
                            h[i] = fmaf(a, h[i], bb);
                            if constexpr (PH2) {
                                if (i & 1) yb = fmaf(Cv[i], h[i], yb);
                                else ya = fmaf(Cv[i], h[i], ya);
                            } else {
                                P[i] *= a;
                            }
                        }
                    }
                    yp[j] = ya + yb;
                }
                if constexpr (PH2) {
                    const float r = reduce_lanes<G>(yp, g);
                    const int t = t0 + g;
                    ys[c * kTS + t] = io<T>::to(fmaf(dsk, uf[c * TSF + t], r));
                }
            }
            // ---- write the stage's outputs
            if constexpr (PH2) {
                __syncthreads();
                T* y = static_cast<T*>(p.y);
                const int nvalid = min(kTS, l_end - l0);
                if (p.vec) {
                    constexpr int VE = 16 / sizeof(T), CPR = kTS / VE;
                    for (int i = tid; i < DT * CPR; i += kThreads) {
                        const int r = i / CPR, ch = i % CPR;
                        if (r < nrows && ch * VE < nvalid)
                            *reinterpret_cast<uint4*>(y + (row0 + r) * (size_t)p.L + l0 + ch * VE) =
                                *reinterpret_cast<const uint4*>(ys + r * kTS + ch * VE);
                    }
                } else {
                    for (int i = tid; i < DT * kTS; i += kThreads) {
                        const int r = i / kTS, t = i % kTS;
                        if (r < nrows && t < nvalid) y[(row0 + r) * (size_t)p.L + l0 + t] = ys[i];
                    }
                }
            }
        }
        cp_async_wait<0>();
        __syncthreads();
    };

    const size_t sfl = (size_t)DT * NP;  // floats of one published state
    const size_t my_off = (size_t)c * NP + (size_t)g * NG;
    if (chunked && chunk > 0) {
        pass(std::false_type{});
        const size_t slot = (size_t)tile * p.n_chunks + chunk;
#pragma unroll
        for (int i = 0; i < NG; ++i) {
            p.aggP[slot * sfl + my_off + i] = P[i];
            p.aggH[slot * sfl + my_off + i] = h[i];
        }
        __threadfence();
        __syncthreads();
        if (tid == 0) st_release(&p.flags[slot], flag_word(gen, kFlagAggregate));
        // Decoupled look-back: walk back until a predecessor's inclusive state is
        // published, then fold the aggregates after it left to right,
        // h <- P_m h + H_m.  Every inclusive state is defined by this same left
        // fold from chunk 0, so the carry is bit-identical whichever predecessor
        // the walk stops at (results do not depend on scheduling).
        int found = -1;
        for (int j = chunk - 1; j >= 0; --j) {
            const size_t sj = (size_t)tile * p.n_chunks + j;
            if (tid == 0) s_misc[0] = wait_flag(&p.flags[sj], gen, p.hdr, (unsigned)tile, (unsigned)j);
            __syncthreads();
            const unsigned kind = s_misc[0];
            __syncthreads();
            if (kind == kFlagInclusive) {
                found = j;
                break;
            }
            if (kind != kFlagAggregate) break;  // wait gave up: error already recorded
        }
        float RH[NG];
#pragma unroll
        for (int i = 0; i < NG; ++i) RH[i] = 0.0f;
        if (found >= 0) {
            const size_t sf = (size_t)tile * p.n_chunks + found;
#pragma unroll
            for (int i = 0; i < NG; ++i) RH[i] = ld_cg(&p.incH[sf * sfl + my_off + i]);
            for (int m = found + 1; m < chunk; ++m) {
                const size_t sm = (size_t)tile * p.n_chunks + m;
#pragma unroll
                for (int i = 0; i < NG; ++i)
                    RH[i] = fmaf(ld_cg(&p.aggP[sm * sfl + my_off + i]), RH[i], ld_cg(&p.aggH[sm * sfl + my_off + i]));
            }
        }
        // inclusive end state of this chunk = P * h_in + H
#pragma unroll
        for (int i = 0; i < NG; ++i) {
            p.incH[slot * sfl + my_off + i] = fmaf(P[i], RH[i], h[i]);
            h[i] = RH[i];
        }
        __threadfence();
        __syncthreads();
        if (tid == 0) st_release(&p.flags[slot], flag_word(gen, kFlagInclusive));
    }

    pass(std::true_type{});

    if (chunked) {
        if (chunk == 0) {
            const size_t slot = (size_t)tile * p.n_chunks;
#pragma unroll
            for (int i = 0; i < NG; ++i) p.incH[slot * sfl + my_off + i] = h[i];
            __threadfence();
            __syncthreads();
            if (tid == 0 && !p.suppress) st_release(&p.flags[slot], flag_word(gen, kFlagInclusive));
        }
        __syncthreads();
        if (tid == 0) finish_launch(p.hdr, (unsigned)(p.n_tiles * p.n_chunks));
    }
}

// ------------------------------------------------------------------ host side

struct KernelInfo {
    const void* fn;
    size_t smem;
    int G;
    int DT;
    int threads;
    int ts;
};

template <typename T, int NP, int G, bool ZOH>
KernelInfo info_for() {
    using LY = Layout<T, NP, G>;
    const void* fn = reinterpret_cast<const void*>(&full_scan_kernel<T, NP, G, ZOH>);
    static std::once_flag once;
    static cudaError_t attr_err = cudaSuccess;
    std::call_once(once, [&] {
        attr_err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)LY::bytes);
    });
    if (attr_err != cudaSuccess) return {nullptr, 0, G, LY::DT, LY::THREADS, LY::TS};
    return {fn, LY::bytes, G, LY::DT, LY::THREADS, LY::TS};
}

template <typename T, bool ZOH>
KernelInfo pick_np(int np) {
    switch (np) {
    case 1: return info_for<T, 1, 1, ZOH>();
    case 2: return info_for<T, 2, 1, ZOH>();
    case 4: return info_for<T, 4, 1, ZOH>();
    case 8: return info_for<T, 8, 2, ZOH>();
    default: return info_for<T, 16, 4, ZOH>();
    }
}

KernelInfo pick(vmb_dtype dt, int np, bool zoh) {
    if (dt == VMB_BF16) return zoh ? pick_np<__nv_bfloat16, true>(np) : pick_np<__nv_bfloat16, false>(np);
    return zoh ? pick_np<float, true>(np) : pick_np<float, false>(np);
}

int pad_states(int N) {
    int np = 1;
    while (np < N) np <<= 1;
    return np;
}

}  // namespace

vmb_status plan_full(const ScanArgs& a, ScanPlan* plan) {
    if (a.N < 1 || a.N > 16) return VMB_ERR_UNSUPPORTED;
    const int np = pad_states(a.N);
    KernelInfo ki = pick(a.dtype, np, (a.flags & VMB_FLAG_B_ZOH) != 0);
    if (!ki.fn) return VMB_ERR_CUDA;
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, ki.fn, ki.threads, ki.smem) != cudaSuccess)
        return VMB_ERR_CUDA;
    if (per_sm < 1) per_sm = 1;
    const long long resident = (long long)per_sm * device_sm_count();
    ScanPlan p{};
    p.np = np;
    p.tile_rows = ki.DT;
    p.tiles_per_bk = (a.D + ki.DT - 1) / ki.DT;
    p.n_seq = a.B * a.K * p.tiles_per_bk;
    // Cut L only when the channel tiles alone cannot fill the GPU; keep chunks
    // at least 128 steps long so the look-back traffic stays small.
    const int kTS = ki.ts;
    int n_chunks = 1;
    if (p.n_seq < resident) {
        const long long want = (resident + p.n_seq - 1) / p.n_seq;
        const long long max_chunks = (a.L + 127) / 128;
        n_chunks = (int)(want < max_chunks ? want : max_chunks);
        if (n_chunks < 1) n_chunks = 1;
    }
    int chunk_len = (a.L + n_chunks - 1) / n_chunks;
    chunk_len = (chunk_len + kTS - 1) / kTS * kTS;
    n_chunks = (a.L + chunk_len - 1) / chunk_len;
    p.n_chunks = n_chunks;
    p.chunk_len = chunk_len;
    p.state_floats = (size_t)ki.DT * np;
    p.ws_bytes = ws_layout(p).total;
    *plan = p;
    return VMB_OK;
}

vmb_status launch_full(const ScanArgs& a, const ScanPlan& plan, cudaStream_t stream) {
    KernelInfo ki = pick(a.dtype, plan.np, (a.flags & VMB_FLAG_B_ZOH) != 0);
    if (!ki.fn) return VMB_ERR_CUDA;
    const size_t es = a.dtype == VMB_BF16 ? 2 : 4;
    FullParams p{};
    p.u = a.u;
    p.dl = a.delta;
    p.A = a.A;
    p.Bs = a.Bs;
    p.Cs = a.Cs;
    p.Dskip = a.Dskip;
    p.bias = a.bias;
    p.y = a.y;
    p.K = a.K;
    p.D = a.D;
    p.N = a.N;
    p.L = a.L;
    p.softplus_on = (a.flags & VMB_FLAG_SOFTPLUS) ? 1 : 0;
    p.tiles_per_bk = plan.tiles_per_bk;
    p.n_tiles = plan.n_seq;
    p.n_chunks = plan.n_chunks;
    p.chunk_len = plan.chunk_len;
    const auto al16 = [](const void* q) { return (reinterpret_cast<uintptr_t>(q) & 15u) == 0; };
    p.vec = ((size_t)a.L * es % 16 == 0) && al16(a.u) && al16(a.delta) && al16(a.Bs) && al16(a.Cs) && al16(a.y);
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
    cudaError_t e = cudaLaunchKernel(ki.fn, dim3(grid), dim3(ki.threads), args, ki.smem, stream);
    return e == cudaSuccess ? VMB_OK : VMB_ERR_CUDA;
}

}  // namespace vmb
