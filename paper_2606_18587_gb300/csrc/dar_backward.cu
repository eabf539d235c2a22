// dar_backward.cu -- host side of the gradients of the causal DAR attention
// forward (Sec. 2.3 training): workspace layout and the launch sequence of
// the kernels in dar_backward.cuh (compiled per storage type in
// dar_backward_f32.cu and, with the tensor-core kernels, dar_backward_tc.cu).
#include "dar_backward.cuh"

namespace dar {
size_t backward_workspace_bytes(dar_dtype dt, int B, int Hq, int Hkv, int N, int dd)
{
    auto al = [](size_t x) { return (x + 255) & ~size_t(255); };
    const size_t es = dt == DAR_F32 ? 4 : 2;
    const size_t qrows = (size_t)B * Hq * N, krows = (size_t)B * Hkv * N;
    return 2 * al(krows * dd * es) + 4 * al(qrows * dd * 4) + 2 * al(qrows * 4) + 2 * al(krows * dd * 4) +
           al((size_t)bwd::kChunks * 4 * Hkv * 64 * dd * 4) + (dt == DAR_BF16 ? 2 * al(qrows * dd * 2) : 0);
}

cudaError_t launch_backward(dar_dtype dt, const BackwardArgs &x, void *workspace, cudaStream_t s)
{
    if (x.B == 0 || x.N == 0)
        return cudaSuccess;
    auto al = [](size_t v) { return (v + 255) & ~size_t(255); };
    const size_t es = dt == DAR_F32 ? 4 : 2;
    const size_t qrows = (size_t)x.B * x.Hq * x.N, krows = (size_t)x.B * x.Hkv * x.N;
    char *p = static_cast<char *>(workspace);
    auto take = [&](size_t n) {
        char *r = p;
        p += al(n);
        return r;
    };
    bwd::Args a;
    a.q = x.q;
    a.k = x.k;
    a.v = x.v;
    a.out = x.out;
    a.dout = x.dout;
    a.Dk = x.Dk;
    a.Uk = x.Uk;
    a.Dv = x.Dv;
    a.Uv = x.Uv;
    a.dq = x.dq;
    a.dk = x.dk;
    a.dv = x.dv;
    a.dDk = x.dDk;
    a.dUk = x.dUk;
    a.dDv = x.dDv;
    a.dUv = x.dUv;
    void *kd = take(krows * x.dd * es), *vd = take(krows * x.dd * es);
    a.kd = kd;
    a.vd = vd;
    a.qt = reinterpret_cast<float *>(take(qrows * x.dd * 4));
    a.dot = reinterpret_cast<float *>(take(qrows * x.dd * 4));
    a.dqt = reinterpret_cast<float *>(take(qrows * x.dd * 4));
    a.od = reinterpret_cast<float *>(take(qrows * x.dd * 4));
    a.drow = reinterpret_cast<float *>(take(qrows * 4));
    a.lse = reinterpret_cast<float *>(take(qrows * 4));
    a.dkd = reinterpret_cast<float *>(take(krows * x.dd * 4));
    a.dvd = reinterpret_cast<float *>(take(krows * x.dd * 4));
    a.part = reinterpret_cast<float *>(take((size_t)bwd::kChunks * 4 * x.Hkv * 64 * x.dd * 4));
    a.qtb = a.dotb = nullptr;
    if (dt == DAR_BF16) {  // bf16 copies of q~ and dO~ for the tensor-core kernels
        a.qtb = reinterpret_cast<bf16 *>(take(qrows * x.dd * 2));
        a.dotb = reinterpret_cast<bf16 *>(take(qrows * x.dd * 2));
    }
    a.B = x.B;
    a.Hq = x.Hq;
    a.Hkv = x.Hkv;
    a.G = x.Hq / x.Hkv;
    a.N = x.N;
    a.w = x.w;
    a.scale = x.scale;
    a.c2 = x.scale * bwd::kLog2e;
    // Eq. 1 as the forward stores it (plain rows of d_down)
    cudaError_t e = launch_down_project_kv(dt, x.dd, x.k, x.v, x.Dk, x.Dv, kd, vd, x.B, x.Hkv, x.N, x.dd, x.dd, -1, s);
    if (e != cudaSuccess)
        return e;
    return dt == DAR_F32 ? bwd::run_f32(x.dd, a, s) : bwd::run_bf16(x.dd, a, s);
}

}  // namespace dar
