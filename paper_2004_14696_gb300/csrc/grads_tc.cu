// Eq. (2) for all n workers with bf16 GEMM operands on the tcgen05 tensor cores.
//
// Same computation as the SIMT pass in grads.cu (forward over the stacked
// M = n B rows, softmax cross entropy, backward with a per-worker weight
// gradient of depth K = B), laid out so that every GEMM has both operands
// K-major, which is what the tcgen05 kernel of gemm_tc.cu consumes:
//
//   forward   Z_l = A_{l-1} . W_l^T          A = act[l-1] [M, in],   B = W_l [out, in]
//   dX        dZ_{l-1} = dZ_l . W_l          A = dZ_l [M, out],      B = W_l^T [in, out]
//   dW        G_i = dZ_l[i]^T . A_{l-1}[i]   A = dZ_l^T [out, M],    B = A_{l-1}^T [in, M]
//                                            (worker i: columns i*B .. i*B+B-1, K = B)
//
// The transposed activations and dZ are written by the epilogue that produces
// them (a store whose 32 lanes cover 32 consecutive samples, 64 contiguous
// bytes), X^T and dZ_L^T by a tiled transpose, W^T by a tiled cast-transpose.
// Leading dimensions are padded to multiples of 8 elements (16 bytes, the TMA
// stride rule); padding is never read (tensor maps carry the logical extents).
#include <math.h>

#include "gemm_tc.cuh"
#include "grads.cuh"

namespace dbw {

namespace {

inline int64_t rup(int64_t x, int64_t m) { return (x + m - 1) / m * m; }

// W_l [out, in] fp32 (rows of length in) -> wb [out, ldw] bf16 and wt [in, ldwt] bf16.
__global__ void cast_transpose_kernel(const float* __restrict__ W, int out, int in, __nv_bfloat16* __restrict__ wb,
                                      int64_t ldw, __nv_bfloat16* __restrict__ wt, int64_t ldwt) {
    __shared__ __nv_bfloat16 tile[32][33];
    const int i0 = blockIdx.x * 32, o0 = blockIdx.y * 32;
    const int tx = threadIdx.x, ty = threadIdx.y;   // 32 x 8
    for (int r = ty; r < 32; r += 8) {
        const int o = o0 + r, i = i0 + tx;
        __nv_bfloat16 v = __float2bfloat16_rn(0.f);
        if (o < out && i < in) {
            v = __float2bfloat16_rn(W[static_cast<int64_t>(o) * in + i]);
            wb[static_cast<int64_t>(o) * ldw + i] = v;
        }
        tile[r][tx] = v;
    }
    __syncthreads();
    for (int r = ty; r < 32; r += 8) {
        const int i = i0 + r, o = o0 + tx;
        if (i < in && o < out) wt[static_cast<int64_t>(i) * ldwt + o] = tile[tx][r];
    }
}

// dst [cols, ldd] = src [rows, lds]^T  (bf16), rows x cols logical.
__global__ void transpose_bf16_kernel(const __nv_bfloat16* __restrict__ src, int rows, int cols, int64_t lds,
                                      __nv_bfloat16* __restrict__ dst, int64_t ldd) {
    __shared__ __nv_bfloat16 tile[32][33];
    const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
    const int tx = threadIdx.x, ty = threadIdx.y;
    for (int r = ty; r < 32; r += 8) {
        const int rr = r0 + r, cc = c0 + tx;
        tile[r][tx] = (rr < rows && cc < cols) ? src[static_cast<int64_t>(rr) * lds + cc] : __float2bfloat16_rn(0.f);
    }
    __syncthreads();
    for (int r = ty; r < 32; r += 8) {
        const int cc = c0 + r, rr = r0 + tx;
        if (cc < cols && rr < rows) dst[static_cast<int64_t>(cc) * ldd + rr] = tile[tx][r];
    }
}

// X[m, :] = bf16(pool[idx[m], :]); an index outside [0, S) reads row 0 (the loss
// kernel poisons that worker).
__global__ void gather_bf16_kernel(const float* __restrict__ pool, int64_t S, int in, const int32_t* __restrict__ idx,
                                   int M, __nv_bfloat16* __restrict__ X, int64_t ldx) {
    for (int m = blockIdx.y; m < M; m += gridDim.y) {
        int64_t r = idx[m];
        if (r < 0 || r >= S) r = 0;
        const float* src = pool + r * in;
        __nv_bfloat16* dst = X + static_cast<int64_t>(m) * ldx;
        for (int c = (blockIdx.x * blockDim.x + threadIdx.x) * 4; c < in; c += gridDim.x * blockDim.x * 4) {
            const float4 v = *reinterpret_cast<const float4*>(src + c);
            __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y), b = __floats2bfloat162_rn(v.z, v.w);
            if (c + 3 < in) {
                *reinterpret_cast<__nv_bfloat162*>(dst + c) = a;
                *reinterpret_cast<__nv_bfloat162*>(dst + c + 2) = b;
            } else {
                for (int e = c; e < in; ++e) dst[e] = __float2bfloat16_rn(src[e]);
            }
        }
    }
}

// Per worker (one CTA): stable log-softmax cross entropy per sample, dZ = (softmax - onehot) / B
// as bf16 into dZ [M, ldz], worker loss = mean of its B sample losses (sample order).
__global__ void __launch_bounds__(256) softmax_xent_ld_kernel(const float* __restrict__ logits, int64_t ldl, int C,
                                                              int B, const int32_t* __restrict__ idx, int64_t S,
                                                              const int32_t* __restrict__ labels,
                                                              float* __restrict__ sample_loss,
                                                              __nv_bfloat16* __restrict__ dZ, int64_t ldz,
                                                              float* __restrict__ loss) {
    const int i = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    __shared__ int bad_s;
    if (threadIdx.x == 0) bad_s = 0;
    __syncthreads();
    const float invB = 1.0f / static_cast<float>(B);
    for (int r = warp; r < B; r += nw) {
        const int64_t row = static_cast<int64_t>(i) * B + r;
        const int64_t sidx = idx[row];
        int y = -1;
        if (sidx >= 0 && sidx < S) y = labels[sidx];
        const bool bad = (y < 0 || y >= C);
        const float* z = logits + row * ldl;
        float mx = -INFINITY;
        for (int c = lane; c < C; c += 32) mx = fmaxf(mx, z[c]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        float se = 0.f;
        for (int c = lane; c < C; c += 32) se += expf(z[c] - mx);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) se += __shfl_xor_sync(0xffffffffu, se, o);
        const float inv_se = 1.0f / se;
        for (int c = lane; c < C; c += 32) {
            float g = expf(z[c] - mx) * inv_se;
            if (c == y) g -= 1.0f;
            dZ[row * ldz + c] = __float2bfloat16_rn(bad ? NAN : g * invB);
        }
        if (lane == 0) {
            sample_loss[row] = bad ? NAN : (mx + logf(se)) - z[y];
            if (bad) bad_s = 1;
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        float acc = 0.f;
        for (int r = 0; r < B; ++r) acc += sample_loss[static_cast<int64_t>(i) * B + r];
        loss[i] = bad_s ? NAN : acc * invB;
    }
}

// G[i, offb + o] = sum_{r < B} dZ[i*B + r, o] (rows in order).
__global__ void bias_grad_ld_kernel(const __nv_bfloat16* __restrict__ dZ, int64_t ldz, int out, int B,
                                    float* __restrict__ G, int64_t ldG, int64_t offb) {
    const int i = blockIdx.y;
    const int o = blockIdx.x * blockDim.x + threadIdx.x;
    if (o >= out) return;
    const __nv_bfloat16* p = dZ + static_cast<int64_t>(i) * B * ldz + o;
    float acc = 0.f;
    for (int r = 0; r < B; ++r) acc += __bfloat162float(p[static_cast<int64_t>(r) * ldz]);
    G[static_cast<int64_t>(i) * ldG + offb + o] = acc;
}

}  // namespace

bool tc_eligible(int prec, int B) { return prec == DBW_PREC_BF16 && B % 32 == 0; }

bool make_tc_plan(int L, const int32_t* widths, int n, int B, TcPlan* P) {
    GradsPlan g;
    if (!make_grads_plan(L, widths, n, B, DBW_PREC_BF16, &g)) return false;
    P->g = g;
    const int64_t M = static_cast<int64_t>(n) * B;
    P->M8 = rup(M, 8);
    int maxw = 0;
    for (int l = 0; l <= L; ++l) maxw = widths[l] > maxw ? widths[l] : maxw;
    size_t cur = 0;
    auto take = [&](size_t bytes) {
        const size_t at = cur;
        cur += (bytes + 255) / 256 * 256;
        return at;
    };
    P->off_status = take(256);
    for (int l = 0; l < L; ++l) {
        const int fin = widths[l], fout = widths[l + 1];
        P->ldw[l] = rup(fin, 8);
        P->ldwt[l] = rup(fout, 8);
        P->off_wb[l] = take(static_cast<size_t>(fout) * P->ldw[l] * 2);
        P->off_wt[l] = take(static_cast<size_t>(fin) * P->ldwt[l] * 2);
    }
    for (int l = 0; l < L; ++l) {   // act[0] = X
        P->ldact[l] = rup(widths[l], 8);
        P->off_act[l] = take(static_cast<size_t>(M) * P->ldact[l] * 2);
        P->off_actT[l] = take(static_cast<size_t>(widths[l]) * P->M8 * 2);
    }
    P->ldlog = rup(widths[L], 4);
    P->off_logits = take(static_cast<size_t>(M) * P->ldlog * 4);
    P->off_sloss = take(static_cast<size_t>(M) * 4);
    P->ldz = rup(maxw, 8);
    P->off_dz[0] = take(static_cast<size_t>(M) * P->ldz * 2);
    P->off_dz[1] = take(static_cast<size_t>(M) * P->ldz * 2);
    P->off_dzT = take(static_cast<size_t>(maxw) * P->M8 * 2);
    P->ws_bytes = cur;
    return true;
}

int worker_grads_tc(const TcPlan& P, const float* w, const float* pool, int64_t S, const int32_t* labels,
                    const int32_t* idx, float* G, int64_t ld, float* loss, char* ws, cudaStream_t st) {
    const GradsPlan& g = P.g;
    const int L = g.L, M = g.M, B = g.B, n = g.n;
    int* status = reinterpret_cast<int*>(ws + P.off_status);
    auto bf = [&](size_t off) { return reinterpret_cast<__nv_bfloat16*>(ws + off); };
    cudaError_t e = cudaMemsetAsync(status, 0, sizeof(int), st);
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_worker_grads: %s", cudaGetErrorString(e));

    // bf16 weights and their transposes
    for (int l = 0; l < L; ++l) {
        const int fin = g.widths[l], fout = g.widths[l + 1];
        dim3 grid((fin + 31) / 32, (fout + 31) / 32);
        cast_transpose_kernel<<<grid, dim3(32, 8), 0, st>>>(w + g.offW[l], fout, fin, bf(P.off_wb[l]), P.ldw[l],
                                                            bf(P.off_wt[l]), P.ldwt[l]);
    }
    // X and X^T
    {
        const int in = g.widths[0];
        dim3 grid((in + 1023) / 1024, M < 65535 ? M : 65535);
        gather_bf16_kernel<<<grid, 256, 0, st>>>(pool, S, in, idx, M, bf(P.off_act[0]), P.ldact[0]);
        dim3 tg((in + 31) / 32, (M + 31) / 32);
        transpose_bf16_kernel<<<tg, dim3(32, 8), 0, st>>>(bf(P.off_act[0]), M, in, P.ldact[0], bf(P.off_actT[0]),
                                                          P.M8);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_worker_grads: %s", cudaGetErrorString(e));

    // forward
    float* logits = reinterpret_cast<float*>(ws + P.off_logits);
    for (int l = 0; l < L; ++l) {
        const int fin = g.widths[l], fout = g.widths[l + 1];
        TcEpi ep{};
        ep.bias = w + g.offb[l];
        int rc;
        if (l < L - 1) {
            ep.out = bf(P.off_act[l + 1]);
            ep.ldo = P.ldact[l + 1];
            ep.outT = bf(P.off_actT[l + 1]);
            ep.ldT = P.M8;
            rc = tc_gemm(TC_HIDDEN, bf(P.off_act[l]), P.ldact[l], M, fin, bf(P.off_wb[l]), P.ldw[l], fout, fin, M,
                         fout, fin, 1, 0, ep, status, st);
        } else {
            ep.outF = logits;
            ep.ldF = P.ldlog;
            rc = tc_gemm(TC_LOGITS, bf(P.off_act[l]), P.ldact[l], M, fin, bf(P.off_wb[l]), P.ldw[l], fout, fin, M,
                         fout, fin, 1, 0, ep, status, st);
        }
        if (rc) return rc;
    }
    // loss, dZ_L and its transpose
    const int C = g.widths[L];
    float* sloss = reinterpret_cast<float*>(ws + P.off_sloss);
    int cur = 0;
    softmax_xent_ld_kernel<<<n, 256, 0, st>>>(logits, P.ldlog, C, B, idx, S, labels, sloss, bf(P.off_dz[0]), P.ldz,
                                              loss);
    {
        dim3 tg((C + 31) / 32, (M + 31) / 32);
        transpose_bf16_kernel<<<tg, dim3(32, 8), 0, st>>>(bf(P.off_dz[0]), M, C, P.ldz, bf(P.off_dzT), P.M8);
    }
    e = cudaGetLastError();
    if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_worker_grads: %s", cudaGetErrorString(e));

    // backward
    for (int l = L - 1; l >= 0; --l) {
        const int fin = g.widths[l], fout = g.widths[l + 1];
        TcEpi ep{};
        ep.G = G;
        ep.ldG = ld;
        ep.off = g.offW[l];
        ep.ldrow = fin;
        int rc = tc_gemm(TC_DW, bf(P.off_dzT), P.M8, fout, M, bf(P.off_actT[l]), P.M8, fin, M, fout, fin, B, n, B,
                         ep, status, st);
        if (rc) return rc;
        bias_grad_ld_kernel<<<dim3((fout + 127) / 128, n), 128, 0, st>>>(bf(P.off_dz[cur]), P.ldz, fout, B, G, ld,
                                                                          g.offb[l]);
        e = cudaGetLastError();
        if (e != cudaSuccess) return fail(DBW_ECUDA, "dbw_worker_grads: %s", cudaGetErrorString(e));
        if (l > 0) {
            TcEpi ex{};
            ex.act = bf(P.off_act[l]);
            ex.ldact = P.ldact[l];
            ex.out = bf(P.off_dz[cur ^ 1]);
            ex.ldo = P.ldz;
            ex.outT = bf(P.off_dzT);
            ex.ldT = P.M8;
            rc = tc_gemm(TC_DX, bf(P.off_dz[cur]), P.ldz, M, fout, bf(P.off_wt[l]), P.ldwt[l], fin, fout, M, fin,
                         fout, 1, 0, ex, status, st);
            if (rc) return rc;
            cur ^= 1;
        }
    }
    return DBW_OK;
}

}  // namespace dbw
