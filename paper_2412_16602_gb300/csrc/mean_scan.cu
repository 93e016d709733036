// mean_scan.cu - VMeanba channel-mean selective scan (Sec. 2.2, Eq. 9) for sm_103a.
//
// y = T^-1(Mamba(T(Abar, Bbar u, C))): T averages the discretised scan inputs
// over the D channels of one (batch, direction), the recurrence runs once on
// the averages, and T^-1 broadcasts its output back to every channel.
//
// One CTA owns one (batch, direction) and one chunk of TC steps; thread (t, s)
// owns step t of the chunk and every S-th channel.
//   A. Channel reduction, fused into the load: each thread reads delta and u of
//      its channels at its step straight from global memory (the lanes of a
//      warp cover consecutive steps, so every load is a coalesced 32-wide row
//      segment), applies the softplus of Eq. 6 once per element, and
//      accumulates sum_d 2^(delta_{d,t} A_{c,n} log2 e) for every state n and
//      sum_d delta_{d,t} u_{d,t}.  Abar is averaged after the exponential
//      (Eq. 9 averages Abar itself); Bbar u = B_n mean_d(delta_d u_d).
//   B. The partial sums of the S channel groups are added in shared memory; the
//      one-channel recurrence runs on the averages in micro-chunks of 8 steps
//      per (state, micro-chunk) thread with a serial combine, a decoupled
//      look-back over the preceding chunks of the same (batch, direction)
//      gives the carry-in state, and ybar_t = sum_n C_{t,n} h_{t,n}.
//   C. Broadcast + skip: y[d, t] = ybar_t + Dskip_c u[d, t] for every channel,
//      coalesced along t (u is read again; it is still in L2).
// The recurrence and the C.h work run once per (b, k) instead of once per
// (b, k, d); the exponentials of Abar stay per (b, k, d, n) because the mean
// is taken after them.
#include <mutex>

#include "vmb_common.cuh"
#include "vmb_internal.h"

namespace vmb {
namespace {

constexpr int kThreads = 256;

__host__ __device__ constexpr size_t a16(size_t v) { return (v + 15) / 16 * 16; }
constexpr int kMC = 8;  // steps per micro-chunk of the local scan

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
    int suppress;
    int bcvec;   // B / C rows 16-byte aligned: async-copied
    int tabvec;  // A, delta_bias, Dskip 16-byte aligned: async-copied
    int no_bcast;  // fused with the cross-merge: no y; ybar (+ the broadcast skip term) only
    int cvec;      // u / y rows allow 4-step vector access (L % 4 == 0, 4-element aligned)
    int bc_group;  // sequences per B / C row block: 1, or G for the grouped basis (K, D are K*G, D/G)
    int gather_h;  // > 0: u is the map x [B, D, H, W] with H = gather_h and u_t its transpose
                   // [B, D, W, H] (K = 4, ybar only): direction k's step l reads the value the
                   // cross-scan would have put there, from x (k = 0, 2) or u_t (k = 1, 3)
    const void* u_t;
    float* save;   // not null: the group means kept for the backward, [n_seq][N + 1][L] fp32
                   // (rows 0 .. N-1 Abar_n, row N the mean of delta u)
    const float* z;    // low-rank Delta (LR kernels): z [n_seq][R][L] fp32 and Wup [K][D][R] fp32,
    const float* Wup;  // delta_raw[d, l] = sum_r Wup[k, d, r] z[r, l] (r in order)
    int R;
    WsHeader* hdr;
    unsigned* flags;
    float* aggP;
    float* aggH;
    float* incH;
};

template <typename T, int NP, int TC, bool ZOH, bool LR = false>
struct MLayout {
    static constexpr int S = kThreads / TC;  // channel groups
    static constexpr int NMC = TC / kMC;
    // channels whose A / bias / Dskip (and, low rank, Wup rows) are staged at a time
    static constexpr int CG = LR ? 128 : 256;
    static constexpr int WR = 8;             // low rank: staged Wup row length (ranks up to 8, zero-padded)
    static constexpr int BCS = TC + 16 / (int)sizeof(T);  // raw B / C row stride (elements), rows 16-byte aligned
    // shared memory, byte offsets
    static constexpr size_t red = 0;                                            // f32 [S][NP][TC] partial sums of Abar
    static constexpr size_t redb = red + (size_t)S * TC * NP * 4;               // f32 [S][NP][TC] of Bbar u (ZOH)
    static constexpr size_t redu = redb + (ZOH ? (size_t)S * TC * NP * 4 : 0);  // f32 [S][TC] sums of delta u
    static constexpr size_t reds = redu + (size_t)S * TC * 4;                   // f32 [S][TC] sums of Dskip u
    static constexpr size_t abar = reds + (size_t)S * TC * 4;                   // f32 [TC][NP]
    static constexpr size_t bubar = abar + (size_t)TC * NP * 4;                 // f32 [TC][NP]
    static constexpr size_t mc = bubar + (size_t)TC * NP * 4;                   // f32 [4][NMC][NP]
    static constexpr size_t ybar = a16(mc + (size_t)4 * NMC * NP * 4);          // f32 [TC], 16-byte aligned
    static constexpr size_t dsu = ybar + (size_t)TC * 4;                        // f32 [TC]
    static constexpr size_t hin = dsu + (size_t)TC * 4;                         // f32 [NP]
    static constexpr size_t bc = a16(hin + (size_t)NP * 4);                     // T [2][NP][BCS] B, C rows as stored
    // channel tables of one group of CG channels: A [CG][NP] (scaled by log2 e
    // in place unless ZOH), delta bias [CG], Dskip [CG]
    static constexpr size_t tab0 = a16(bc + (size_t)2 * NP * BCS * sizeof(T));
    static constexpr size_t tab_bytes = (size_t)CG * NP * 4 + 2 * (size_t)CG * 4 + (LR ? (size_t)CG * WR * 4 : 0);
    static constexpr size_t bytes1 = tab0 + tab_bytes;
    static constexpr size_t bytes2 = bytes1;
    static_assert(kThreads % TC == 0 && TC % 32 == 0, "a warp covers 32 consecutive steps");
    static_assert(NP * NMC <= kThreads, "local scan mapping");
    static_assert(bytes2 <= 110 * 1024, "mean-scan tile must leave room for two CTAs per SM");
};

// Stage group g0 of the channel tables (raw A rows, delta bias, Dskip) into
// buffer `tb`: 16-byte async copies where rows are aligned, element loads
// otherwise; channels past the group are zero.
template <typename T, int NP, int TC, bool ZOH, bool LR = false>
__device__ __forceinline__ void stage_tables(const MeanParams& p, unsigned char* tb, int k, int g0, int gn) {
    using LY = MLayout<T, NP, TC, ZOH, LR>;
    constexpr int CG = LY::CG;
    float* ta = reinterpret_cast<float*>(tb);
    float* tbias = ta + CG * NP;
    float* tdsk = tbias + CG;
    const int tid = threadIdx.x;
    const float* Ag = p.A + ((size_t)k * p.D + g0) * p.N;
    bool rows_done = false;
    if constexpr (NP % 4 == 0) {
        if (p.N == NP && p.tabvec) {
            for (int i = tid; i < CG * NP / 4; i += kThreads) {
                const int r = i / (NP / 4);
                const bool ok = r < gn;
                cp_async16(ta + 4 * i, ok ? Ag + 4 * i : p.A, ok ? 16 : 0);
            }
            rows_done = true;
        }
    }
    if (!rows_done) {
        for (int i = tid; i < CG * NP; i += kThreads) {
            const int r = i / NP, n = i % NP;
            ta[i] = (r < gn && n < p.N) ? __ldg(Ag + (size_t)r * p.N + n) : 0.0f;
        }
    }
    const float* bg = p.bias + (size_t)k * p.D + g0;
    const float* dg = p.Dskip + (size_t)k * p.D + g0;
    if (p.tabvec && (((size_t)k * p.D + g0) & 3) == 0) {
        for (int i = tid; i < 2 * CG / 4; i += kThreads) {
            const int which = i / (CG / 4), r = 4 * (i % (CG / 4));
            const int nb = max(0, min(4, gn - r)) * 4;
            cp_async16((which ? tdsk : tbias) + r, nb ? (which ? dg : bg) + r : p.bias, nb);
        }
    } else {
        for (int i = tid; i < CG; i += kThreads) {
            tbias[i] = i < gn ? __ldg(bg + i) : 0.0f;
            tdsk[i] = i < gn ? __ldg(dg + i) : 0.0f;
        }
    }
    if constexpr (LR) {
        // Wup rows of the group, [CG][WR] fp32, zero past R and past the group
        float* tw = reinterpret_cast<float*>(tb) + CG * NP + 2 * CG;
        const float* wg = p.Wup + ((size_t)k * p.D + g0) * p.R;
        for (int i = tid; i < CG * LY::WR; i += kThreads) {
            const int r = i / LY::WR, q = i % LY::WR;
            tw[i] = (r < gn && q < p.R) ? __ldg(wg + (size_t)r * p.R + q) : 0.0f;
        }
    }
}

// Four consecutive elements with an L2 eviction policy (16 bytes fp32, 8 bytes bf16).
__device__ __forceinline__ void ld4_hint(const float* q, uint64_t pol, float (&v)[4]) {
    asm volatile("ld.global.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], %5;"
                 : "=f"(v[0]), "=f"(v[1]), "=f"(v[2]), "=f"(v[3])
                 : "l"(q), "l"(pol));
}
__device__ __forceinline__ void ld4_hint(const __nv_bfloat16* q, uint64_t pol, float (&v)[4]) {
    unsigned a, b;
    asm volatile("ld.global.L2::cache_hint.v2.b32 {%0, %1}, [%2], %3;" : "=r"(a), "=r"(b) : "l"(q), "l"(pol));
    v[0] = __uint_as_float(a << 16);
    v[1] = __uint_as_float(a & 0xffff0000u);
    v[2] = __uint_as_float(b << 16);
    v[3] = __uint_as_float(b & 0xffff0000u);
}
__device__ __forceinline__ void st4_hint(float* q, const float (&v)[4], uint64_t pol) {
    asm volatile("st.global.L2::cache_hint.v4.f32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(q), "f"(v[0]), "f"(v[1]),
                 "f"(v[2]), "f"(v[3]), "l"(pol)
                 : "memory");
}
__device__ __forceinline__ void st4_hint(__nv_bfloat16* q, const float (&v)[4], uint64_t pol) {
    const unsigned a = __bfloat16_as_ushort(__float2bfloat16_rn(v[0])) |
                       ((unsigned)__bfloat16_as_ushort(__float2bfloat16_rn(v[1])) << 16);
    const unsigned b = __bfloat16_as_ushort(__float2bfloat16_rn(v[2])) |
                       ((unsigned)__bfloat16_as_ushort(__float2bfloat16_rn(v[3])) << 16);
    asm volatile("st.global.L2::cache_hint.v2.b32 [%0], {%1, %2}, %3;" ::"l"(q), "r"(a), "r"(b), "l"(pol) : "memory");
}

// LR: the raw Deltas are formed from the low-rank form of Eq. 6 (z, Wup) at
// the thread's step instead of being read: R FMAs per channel, r in order (the
// selection kernel's epilogue order, so fp32 results are bit-identical to
// selection -> raw Deltas -> this scan), z of the step in registers, the Wup
// row read through L1 (every lane of a warp has the same channel).
constexpr int kLRMax = 8;  // ranks the LR kernels hold in registers

template <typename T, int NP, int TC, bool ZOH, bool LR = false>
__global__ void __launch_bounds__(kThreads, ZOH ? 2 : 3) mean_scan_kernel(const MeanParams p) {
    using LY = MLayout<T, NP, TC, ZOH, LR>;
    constexpr int S = LY::S, NMC = LY::NMC, CG = LY::CG, BCS = LY::BCS;
    extern __shared__ __align__(16) unsigned char smb[];
    float* red = reinterpret_cast<float*>(smb + LY::red);
    float* redb = reinterpret_cast<float*>(smb + LY::redb);
    float* redu = reinterpret_cast<float*>(smb + LY::redu);
    float* reds = reinterpret_cast<float*>(smb + LY::reds);
    float* abar = reinterpret_cast<float*>(smb + LY::abar);
    float* bubar = reinterpret_cast<float*>(smb + LY::bubar);
    float* mcP = reinterpret_cast<float*>(smb + LY::mc);
    float* mcH = mcP + NMC * NP;
    float* exP = mcH + NMC * NP;
    float* exH = exP + NMC * NP;
    float* s_ybar = reinterpret_cast<float*>(smb + LY::ybar);
    float* s_dsu = reinterpret_cast<float*>(smb + LY::dsu);
    float* s_hin = reinterpret_cast<float*>(smb + LY::hin);
    T* sB = reinterpret_cast<T*>(smb + LY::bc);
    T* sC = sB + NP * BCS;
    __shared__ unsigned s_misc[2];
    __shared__ unsigned s_scr[2 * kThreads / 32 + 2];

    pdl_wait();
    pdl_launch_dependents();
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
    const size_t bcrow0 = (size_t)(seq / p.bc_group) * N;  // first row of Bs/Cs
    const T* u = static_cast<const T*>(p.u);
    const T* dlr = static_cast<const T*>(p.dl);

    // ---------------------------------------------------------------- prologue
    // B and C of the chunk as stored ([n][t] rows, zero past the problem) and the
    // first group's channel tables go in flight as async copies; the first
    // delta / u values of phase A are requested before anything waits.
    {
        const T* Bs = static_cast<const T*>(p.Bs);
        const T* Cs = static_cast<const T*>(p.Cs);
        if (p.bcvec) {
            constexpr int VE = 16 / (int)sizeof(T), CPR = TC / VE;
            for (int i = tid; i < 2 * NP * CPR; i += kThreads) {
                const int which = i / (NP * CPR), r = (i / CPR) % NP, ch = i % CPR;
                const bool ok = r < N && ch * VE < nvalid;
                const T* src = (which ? Cs : Bs) + (bcrow0 + r) * (size_t)L + l0 + ch * VE;
                cp_async16((which ? sC : sB) + r * BCS + ch * VE, ok ? src : Bs, ok ? 16 : 0);
            }
        } else {
            for (int i = tid; i < 2 * NP * TC; i += kThreads) {
                const int which = i / (NP * TC), r = (i / TC) % NP, t = i % TC;
                T v = T(0.0f);
                if (r < N && t < nvalid) v = (which ? Cs : Bs)[(bcrow0 + r) * (size_t)L + l0 + t];
                (which ? sC : sB)[r * BCS + t] = v;
            }
        }
    }
    const int ngroups = (D + CG - 1) / CG;
    stage_tables<T, NP, TC, ZOH, LR>(p, smb + LY::tab0, k, 0, min(CG, D));
    cp_async_commit();

    // ---------------------------------------------------------------- phase A
    const int rt = tid % TC;  // step of this thread
    const int sg = tid / TC;  // channel group of this thread
    const bool tv = rt < nvalid;
    float acc[NP], accb[NP];
#pragma unroll
    for (int n = 0; n < NP; ++n) {
        acc[n] = 0.0f;
        accb[n] = 0.0f;
    }
    float sdu = 0.0f, sdsu = 0.0f;
    // Channel groups of CG: the group's A, bias and Dskip are in shared memory
    // (async copies, the first group's issued with the prologue), A is scaled by
    // log2 e in place once it lands, then every thread reduces its channels of
    // the group with the delta and u of the next kPF channels already in flight.
    // Six channels ahead with 16 states and 128-step chunks (measured on GB300
    // at batch 128 and on the batch-32 stage-1 map: 4-5% faster than 4 or 8,
    // and fewer spills at 80 registers), eight otherwise (7% faster than six
    // with one state).
    constexpr int kPF = (NP >= 16 && TC >= 128) ? 6 : 8;
    const size_t col = (size_t)l0 + (tv ? rt : 0);
    const T* dcol = dlr + urow0 * (size_t)L + col;
    const T* ucol = u + urow0 * (size_t)L + col;
    if (p.gather_h > 0) {
        // the value the App. A cross-scan puts at step l of direction k: 0 reads
        // the (b, d) plane of x row by row, 1 column by column (the rows of its
        // transpose u_t), 2 and 3 the same in reverse; the planes have the same
        // channel stride L as the rows of u
        const int lr = (k >= 2) ? L - 1 - (int)col : (int)col;
        ucol = ((k & 1) ? static_cast<const T*>(p.u_t) : u) + (size_t)(seq / p.K) * D * (size_t)L + lr;
    }
    // u is read again by the broadcast pass: keep it in L2; delta streams through
    const uint64_t keep = l2_evict_last(), stream = l2_evict_first();
    float* s_a2 = reinterpret_cast<float*>(smb + LY::tab0);
    const float* s_bias = s_a2 + CG * NP;
    const float* s_dsk = s_bias + CG;
    const float* s_wup = s_dsk + CG;  // low rank: the group's Wup rows [CG][WR]
    // Offsets within the (b, k) slab are 32-bit (D * L < 2^31, checked by the
    // planner); a thread's consecutive channels are SL elements apart.
    const int SL = S * L;
    float vd[kPF], vu[kPF];
    float zr[LR ? kLRMax : 1];  // LR: z of this thread's step
    if constexpr (LR) {
#pragma unroll
        for (int r = 0; r < kLRMax; ++r)
            zr[r] = (tv && r < p.R) ? __ldg(p.z + ((size_t)seq * p.R + r) * L + col) : 0.0f;
    }
    static_assert(!LR || kLRMax == 8, "the staged Wup rows hold 8 ranks");
    {
        // the first group's first channels, requested before the tables are waited on
        const int gn = min(CG, D);
        int o = sg * L;
#pragma unroll
        for (int q = 0; q < kPF; ++q, o += SL) {
            const int d = sg + q * S;
            vd[q] = (!LR && tv && d < gn) ? ld_hint(dcol + o, stream) : 0.0f;
            vu[q] = (tv && d < gn) ? ld_hint(ucol + o, keep) : 0.0f;
        }
    }
    // one channel's contribution: softplus, the N exponentials of Abar, delta u
    auto reduce_one = [&](float vdq, float vuq, int d) {
        if constexpr (LR) {
            // the row is zero past R, as is zr: the padded terms add exact zeros
            const float4* w4 = reinterpret_cast<const float4*>(s_wup + d * LY::WR);
            const float4 wa = w4[0], wb = w4[1];
            float rs = 0.0f;
            rs = fmaf(wa.x, zr[0], rs);
            rs = fmaf(wa.y, zr[1], rs);
            rs = fmaf(wa.z, zr[2], rs);
            rs = fmaf(wa.w, zr[3], rs);
            rs = fmaf(wb.x, zr[4], rs);
            rs = fmaf(wb.y, zr[5], rs);
            rs = fmaf(wb.z, zr[6], rs);
            rs = fmaf(wb.w, zr[7], rs);
            vdq = rs;
        }
        const float v = vdq + s_bias[d];
        const float dv = p.softplus_on ? softplus(v) : v;
        const float* a2 = s_a2 + d * NP;  // broadcast reads: every lane has the same d
        if constexpr (ZOH) {
#pragma unroll
            for (int n = 0; n < NP; ++n) {
                const float an = a2[n];
                const float em1 = expm1f(dv * an);
                acc[n] += 1.0f + em1;
                accb[n] = fmaf(an != 0.0f ? em1 / an : dv, vuq, accb[n]);
            }
        } else if constexpr (NP % 4 == 0) {
#pragma unroll
            for (int n = 0; n < NP; n += 4) {
                const float4 qa = *reinterpret_cast<const float4*>(a2 + n);
                if constexpr (TC >= 64) {
                    // packed f32x2 products and sums: half the issue slots (measured
                    // 4-5% faster on the large maps that take these chunk lengths)
                    const float2 dv2 = make_float2(dv, dv);
                    const float2 t01 = __fmul2_rn(dv2, make_float2(qa.x, qa.y));
                    const float2 t23 = __fmul2_rn(dv2, make_float2(qa.z, qa.w));
                    const float2 a01 = __fadd2_rn(make_float2(acc[n], acc[n + 1]), make_float2(ex2(t01.x), ex2(t01.y)));
                    const float2 a23 = __fadd2_rn(make_float2(acc[n + 2], acc[n + 3]), make_float2(ex2(t23.x), ex2(t23.y)));
                    acc[n] = a01.x;
                    acc[n + 1] = a01.y;
                    acc[n + 2] = a23.x;
                    acc[n + 3] = a23.y;
                } else {
                    acc[n] += ex2(dv * qa.x);
                    acc[n + 1] += ex2(dv * qa.y);
                    acc[n + 2] += ex2(dv * qa.z);
                    acc[n + 3] += ex2(dv * qa.w);
                }
            }
        } else {
#pragma unroll
            for (int n = 0; n < NP; ++n) acc[n] += ex2(dv * a2[n]);
        }
        sdu = fmaf(dv, vuq, sdu);
        if (p.skip_mean) sdsu = fmaf(s_dsk[d], vuq, sdsu);
    };
    for (int gi = 0; gi < ngroups; ++gi) {
        const int g0 = gi * CG, gn = min(CG, D - g0);
        if (gi > 0) {
            __syncthreads();  // the previous group's tables are no longer read
            stage_tables<T, NP, TC, ZOH, LR>(p, smb + LY::tab0, k, g0, gn);
            cp_async_commit();
        }
        cp_async_wait<0>();
        __syncthreads();  // this group's tables have landed
        if constexpr (!ZOH) {
            for (int i = tid; i < CG * NP; i += kThreads) s_a2[i] *= kLog2e;
            __syncthreads();
        }
        if (!tv) continue;
        if (gi > 0) {
            int o = (g0 + sg) * L;
#pragma unroll
            for (int q = 0; q < kPF; ++q, o += SL) {
                const int d = sg + q * S;
                vd[q] = (!LR && d < gn) ? ld_hint(dcol + o, stream) : 0.0f;
                vu[q] = d < gn ? ld_hint(ucol + o, keep) : 0.0f;
            }
        }
        for (int d0 = sg; d0 < gn; d0 += kPF * S) {
            float nd[kPF], nu[kPF];
            int o = (g0 + d0 + kPF * S) * L;  // the next batch's first channel
            if (d0 + (2 * kPF - 1) * S < gn) {
                // the next batch is entirely in range: no per-channel checks
#pragma unroll
                for (int q = 0; q < kPF; ++q, o += SL) {
                    nd[q] = LR ? 0.0f : ld_hint(dcol + o, stream);
                    nu[q] = ld_hint(ucol + o, keep);
                }
            } else {
#pragma unroll
                for (int q = 0; q < kPF; ++q, o += SL) {
                    const int d = d0 + (q + kPF) * S;
                    nd[q] = (!LR && d < gn) ? ld_hint(dcol + o, stream) : 0.0f;
                    nu[q] = d < gn ? ld_hint(ucol + o, keep) : 0.0f;
                }
            }
            if (d0 + (kPF - 1) * S < gn) {
#pragma unroll
                for (int q = 0; q < kPF; ++q) reduce_one(vd[q], vu[q], d0 + q * S);
            } else {
#pragma unroll
                for (int q = 0; q < kPF; ++q) {
                    const int d = d0 + q * S;
                    if (d >= gn) break;
                    reduce_one(vd[q], vu[q], d);
                }
            }
#pragma unroll
            for (int q = 0; q < kPF; ++q) {
                vd[q] = nd[q];
                vu[q] = nu[q];
            }
        }
    }
    if (!tv) {
        // steps past the end of the sequence: identity (Abar = 1, Bbar u = 0)
#pragma unroll
        for (int n = 0; n < NP; ++n) acc[n] = sg == 0 ? (float)D : 0.0f;
    }

    // ---------------------------------------------------------------- phase B
#pragma unroll
    for (int n = 0; n < NP; ++n) {  // [S][NP][TC]: lanes (consecutive t) hit consecutive banks
        red[(sg * NP + n) * TC + rt] = acc[n];
        if constexpr (ZOH) redb[(sg * NP + n) * TC + rt] = accb[n];
    }
    redu[sg * TC + rt] = sdu;
    reds[sg * TC + rt] = sdsu;
    __syncthreads();
    const float invD = 1.0f / (float)D;
    for (int i = tid; i < TC * NP; i += kThreads) {
        const int n = i / TC, t = i % TC;
        float sa = 0.0f, sb = 0.0f, su = 0.0f;
#pragma unroll
        for (int s2 = 0; s2 < S; ++s2) {
            sa += red[(s2 * NP + n) * TC + t];
            if constexpr (ZOH) sb += redb[(s2 * NP + n) * TC + t];
            su += redu[s2 * TC + t];
        }
        abar[t * NP + n] = sa * invD;
        bubar[t * NP + n] = io<T>::cvt(sB[n * BCS + t]) * (ZOH ? sb : su) * invD;
        if (p.save && t < nvalid) {
            float* sv = p.save + (size_t)seq * (N + 1) * L + l0 + t;
            if (n < N) sv[(size_t)n * L] = sa * invD;
            if (n == 0) sv[(size_t)N * L] = su * invD;
        }
    }
    for (int t = tid; t < TC; t += kThreads) {
        float sd = 0.0f;
#pragma unroll
        for (int s2 = 0; s2 < S; ++s2) sd += reds[s2 * TC + t];
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
    }
    __syncthreads();
    if (chunked) {
        const size_t slot = (size_t)seq * p.n_chunks + chunk;
        if (tid == 0 && !(p.suppress && chunk == 0))
            st_release(&p.flags[slot], flag_word(gen, chunk == 0 ? kFlagInclusive : kFlagAggregate));
        float RH = 0.0f;
        if (chunk > 0) {
            // Decoupled look-back (the whole block polls 256 predecessors per round)
            // with a left fold after the inclusive state found: the carry is
            // bit-identical whichever predecessor the walk stops at.
            const int found = lookback_find_block<kThreads>(p.flags + (size_t)seq * p.n_chunks, chunk, gen, p.hdr,
                                                            (unsigned)seq, s_scr);
            if (found >= 0) {
                // Fold the aggregates after the inclusive state left to right.  They are
                // staged into shared memory (the partial-sum area, free by now) in
                // batches with all loads in flight at once, then folded from there.
                constexpr int kFB = (S * TC * NP) / (2 * NP);  // aggregates per batch
                float* sP = red;
                float* sH = red + kFB * NP;
                if (tid < NP) RH = ld_cg(&p.incH[((size_t)seq * p.n_chunks + found) * NP + tid]);
                for (int m0 = found + 1; m0 < chunk; m0 += kFB) {
                    const int nb = min(kFB, chunk - m0);
                    for (int i = tid; i < nb * NP; i += kThreads) {
                        const size_t smi = (size_t)seq * p.n_chunks + m0 + i / NP;
                        sP[i] = ld_cg(&p.aggP[smi * NP + i % NP]);
                        sH[i] = ld_cg(&p.aggH[smi * NP + i % NP]);
                    }
                    __syncthreads();
                    if (tid < NP) {
#pragma unroll 8
                        for (int q = 0; q < nb; ++q) RH = fmaf(sP[q * NP + tid], RH, sH[q * NP + tid]);
                    }
                    __syncthreads();
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
            abar[t * NP + n] = io<T>::cvt(sC[n * BCS + t]) * h;
        }
    }
    __syncthreads();
    for (int t = tid; t < TC; t += kThreads) {
        float s2 = 0.0f;
#pragma unroll
        for (int n = 0; n < NP; ++n) s2 += abar[t * NP + n];
        s_ybar[t] = s2;
        // fused with the merge, ybar carries the broadcast skip term (the same
        // fp32 add the broadcast below would do)
        if (p.ybar && t < nvalid) p.ybar[(size_t)seq * L + l0 + t] = (p.no_bcast && p.skip_mean) ? s2 + s_dsu[t] : s2;
    }
    __syncthreads();

    // ---------------------------------------------------------------- phase C
    if (!p.no_bcast && p.cvec) {
        // thread (quad, channel group): four consecutive steps of every DG-th
        // channel, 128-bit (bf16: 64-bit) loads and stores
        constexpr int Q = TC / 4, DG = kThreads / Q;
        const int t4 = 4 * (tid % Q), dg = tid / Q;
        if (t4 < nvalid) {
            const bool qfull = t4 + 4 <= nvalid;
            T* yc = static_cast<T*>(p.y) + urow0 * (size_t)L + l0 + t4;
            const T* uc = u + urow0 * (size_t)L + l0 + t4;
            const float4 yq = *reinterpret_cast<const float4*>(s_ybar + t4);
            const float yb[4] = {yq.x, yq.y, yq.z, yq.w};
            const uint64_t ev = l2_evict_first();
            const int SLg = DG * L;
            if (p.skip_mean) {
                float yv[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) yv[j] = yb[j] + s_dsu[t4 + j];
                int o = dg * L;
                for (int d = dg; d < D; d += DG, o += SLg) {
                    if (qfull) {
                        st4_hint(yc + o, yv, ev);
                    } else {
                        for (int j = 0; j < nvalid - t4; ++j) st_hint(yc + o + j, yv[j], ev);
                    }
                }
            } else {
                constexpr int kPC = 8;
                const bool dsk_smem = ngroups == 1;
                const float* dsk_g = p.Dskip + (size_t)k * D;
                for (int d0 = dg; d0 < D; d0 += kPC * DG) {
                    float uv[kPC][4];
                    int o = d0 * L;
#pragma unroll
                    for (int q = 0; q < kPC; ++q, o += SLg) {
                        const int d = d0 + q * DG;
                        if (d < D && qfull) {
                            ld4_hint(uc + o, ev, uv[q]);
                        } else {
#pragma unroll
                            for (int j = 0; j < 4; ++j) uv[q][j] = (d < D && t4 + j < nvalid) ? ld_hint(uc + o + j, ev) : 0.0f;
                        }
                    }
                    o = d0 * L;
#pragma unroll
                    for (int q = 0; q < kPC; ++q, o += SLg) {
                        const int d = d0 + q * DG;
                        if (d >= D) break;
                        const float dk = dsk_smem ? s_dsk[d] : __ldg(dsk_g + d);
                        float yv[4];
#pragma unroll
                        for (int j = 0; j < 4; ++j) yv[j] = fmaf(dk, uv[q][j], yb[j]);  // as the fused merge does
                        if (qfull) {
                            st4_hint(yc + o, yv, ev);
                        } else {
                            for (int j = 0; j < nvalid - t4; ++j) st_hint(yc + o + j, yv[j], ev);
                        }
                    }
                }
            }
        }
    } else if (tv && !p.no_bcast) {
        T* yc = static_cast<T*>(p.y) + urow0 * (size_t)L + l0 + rt;
        const T* uc = u + urow0 * (size_t)L + l0 + rt;
        const float yb = s_ybar[rt];
        const uint64_t ev = l2_evict_first();
        if (p.skip_mean) {
            // y = ybar + the mean skip term: one value for every channel
            const float yv = yb + s_dsu[rt];
            int o = sg * L;
            for (int d = sg; d < D; d += S, o += SL) st_hint(yc + o, yv, ev);
        } else {
            // y = ybar + Dskip u as one FMA (the fused merge does the same); with
            // short chunks (many channels per thread) all of a thread's channels
            // of a 192-channel map are in flight in one round
            constexpr int kPC = TC == 32 ? 24 : 8;
            const bool dsk_smem = ngroups == 1;  // Dskip of every channel is still staged
            const float* dsk_g = p.Dskip + (size_t)k * D;
            for (int d0 = sg; d0 < D; d0 += kPC * S) {
                float uv[kPC];
                const bool full = d0 + (kPC - 1) * S < D;
                int o = d0 * L;
#pragma unroll
                for (int q = 0; q < kPC; ++q, o += SL)
                    uv[q] = (full || d0 + q * S < D) ? ld_hint(uc + o, ev) : 0.0f;
                o = d0 * L;
#pragma unroll
                for (int q = 0; q < kPC; ++q, o += SL) {
                    const int d = d0 + q * S;
                    if (!full && d >= D) break;
                    const float dk = dsk_smem ? s_dsk[d] : __ldg(dsk_g + d);
                    st_hint(yc + o, fmaf(dk, uv[q], yb), ev);
                }
            }
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
    size_t smem;   // D <= 256: one buffer of channel tables
    size_t smem2;  // D > 256: two
};

template <typename T, int NP, int TC, bool ZOH, bool LR>
KInfo minfo() {
    using LY = MLayout<T, NP, TC, ZOH, LR>;
    const void* fn = reinterpret_cast<const void*>(&mean_scan_kernel<T, NP, TC, ZOH, LR>);
    static std::once_flag once;
    static cudaError_t err = cudaSuccess;
    std::call_once(once, [&] {
        err = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)LY::bytes2);
    });
    if (err != cudaSuccess) return {nullptr, 0, 0};
    return {fn, LY::bytes1, LY::bytes2};
}

template <typename T, int NP, bool ZOH, bool LR>
KInfo pick_tc(int tc) {
    switch (tc) {
    case 32: return minfo<T, NP, 32, ZOH, LR>();
    case 128: return minfo<T, NP, 128, ZOH, LR>();
    default: return minfo<T, NP, 64, ZOH, LR>();
    }
}

template <typename T, bool ZOH, bool LR>
KInfo pick_np(int np, int tc) {
    switch (np) {
    case 1: return pick_tc<T, 1, ZOH, LR>(tc);
    case 2: return pick_tc<T, 2, ZOH, LR>(tc);
    case 4: return pick_tc<T, 4, ZOH, LR>(tc);
    case 8: return pick_tc<T, 8, ZOH, LR>(tc);
    default: return pick_tc<T, 16, ZOH, LR>(tc);
    }
}

// lr: the low-rank-Delta kernels (Euler Bbar only)
KInfo mpick(vmb_dtype dt, int np, int tc, bool zoh, bool lr = false) {
    if (lr) return dt == VMB_BF16 ? pick_np<__nv_bfloat16, false, true>(np, tc) : pick_np<float, false, true>(np, tc);
    if (dt == VMB_BF16)
        return zoh ? pick_np<__nv_bfloat16, true, false>(np, tc) : pick_np<__nv_bfloat16, false, false>(np, tc);
    return zoh ? pick_np<float, true, false>(np, tc) : pick_np<float, false, false>(np, tc);
}

}  // namespace

vmb_status plan_mean(const ScanArgs& a, ScanPlan* plan) {
    if (a.N < 1 || a.N > 16) return VMB_ERR_UNSUPPORTED;
    if ((long long)a.D * a.L >= (1LL << 31)) return VMB_ERR_UNSUPPORTED;  // 32-bit offsets within a (b, k) slab
    int np = 1;
    while (np < a.N) np <<= 1;
    const bool zoh = (a.flags & VMB_FLAG_B_ZOH) != 0;
    // Longest chunk whose grid still fills the GPU (one CTA per (b, k, chunk)):
    // two waves of CTAs when a sequence has many channels (each CTA stages its
    // channels' tables and reduces D channels per step), 0.8 of a wave when it
    // has at most 256 (there a longer chunk amortises the fixed work of a CTA;
    // measured on GB300 over batch 1 to 4 stage-1 maps, the batch-32 stages and
    // grouped-basis views).  The tests can force a chunk length (vmb_testing.h).
    const long long seqs = (long long)a.B * a.K;
    int tc = 32;
    const int forced = forced_mean_chunk();
    for (int cand : {128, 64, 32}) {
        if (forced && cand != forced) continue;
        KInfo ki = mpick(a.dtype, np, cand, zoh);
        if (!ki.fn) return VMB_ERR_CUDA;
        int per_sm = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, ki.fn, kThreads, a.D > 256 ? ki.smem2 : ki.smem) !=
            cudaSuccess)
            return VMB_ERR_CUDA;
        const long long resident = (long long)(per_sm < 1 ? 1 : per_sm) * device_sm_count();
        const long long ctas = seqs * ((a.L + cand - 1) / cand);
        const bool fills = a.D <= 256 ? 5 * ctas >= 4 * resident : ctas >= 2 * resident;
        if (forced || fills || cand == 32) {
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
    const bool lr = a.R > 0;
    if (lr && ((a.flags & VMB_FLAG_B_ZOH) || a.R > kLRMax || a.bc_group != 1)) return VMB_ERR_UNSUPPORTED;
    KInfo ki = mpick(a.dtype, plan.np, plan.chunk_len, (a.flags & VMB_FLAG_B_ZOH) != 0, lr);
    if (!ki.fn) return VMB_ERR_CUDA;
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
    p.suppress = (a.flags & VMB_FLAG_TEST_SUPPRESS_PUBLISH) ? 1 : 0;
    const size_t es = a.dtype == VMB_BF16 ? 2 : 4;
    const auto al16 = [](const void* q) { return (reinterpret_cast<uintptr_t>(q) & 15u) == 0; };
    p.bcvec = ((size_t)a.L * es % 16 == 0) && al16(a.Bs) && al16(a.Cs);
    const auto al4e = [&](const void* q) { return (reinterpret_cast<uintptr_t>(q) % (4 * es)) == 0; };
    p.cvec = (a.L % 4 == 0) && al4e(a.u) && (a.y == nullptr || al4e(a.y));
    p.no_bcast = a.no_bcast ? 1 : 0;
    p.bc_group = a.bc_group;
    p.gather_h = a.gather_h;
    p.u_t = a.u_t;
    p.save = a.saved;
    p.z = lr ? static_cast<const float*>(a.delta) : nullptr;
    p.Wup = a.Wup;
    p.R = a.R;
    p.tabvec = al16(a.A) && al16(a.bias) && al16(a.Dskip);
    const WsLayout w = ws_layout(plan);
    unsigned char* ws = static_cast<unsigned char*>(a.ws);
    p.hdr = reinterpret_cast<WsHeader*>(ws);
    p.flags = reinterpret_cast<unsigned*>(ws + w.flags_off);
    p.aggP = reinterpret_cast<float*>(ws + w.aggP_off);
    p.aggH = reinterpret_cast<float*>(ws + w.aggH_off);
    p.incH = reinterpret_cast<float*>(ws + w.incH_off);
    const unsigned grid = (unsigned)(plan.n_seq * plan.n_chunks);
    void* args[] = {&p};
    cudaError_t e = launch_kernel(ki.fn, dim3(grid), dim3(kThreads), a.D > 256 ? ki.smem2 : ki.smem, args, stream);
    return e == cudaSuccess ? VMB_OK : VMB_ERR_CUDA;
}

}  // namespace vmb
