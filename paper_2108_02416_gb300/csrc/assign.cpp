// Host side of libaspis: the subset-based file assignment (Algorithm 2) and
// the small helpers shared by the entry points.
#include <cstdlib>
#include <cstring>
#include <vector>

#include "aspis.h"

namespace {

int64_t choose(int n, int k)
{
    if (k < 0 || k > n) return 0;
    if (k > n - k) k = n - k;
    int64_t c = 1;
    for (int i = 0; i < k; ++i) c = c * (n - i) / (i + 1);
    return c;
}

// Depth-first generation of the r-subsets of {0..K-1}: the recursion visits
// the smallest available worker first at each depth, so subsets come out in
// lexicographic order and subset number i is file i (Algorithm 2; Example 1:
// file 0 is {0,...,r-1}).
struct SubsetWriter {
    int K, r;
    uint8_t *out;
    int64_t next = 0;
    uint8_t cur[ASPIS_MAX_R];

    void walk(int depth, int first)
    {
        if (depth == r) {
            std::memcpy(out + next * r, cur, (size_t)r);
            ++next;
            return;
        }
        for (int w = first; w <= K - (r - depth); ++w) {
            cur[depth] = (uint8_t)w;
            walk(depth + 1, w + 1);
        }
    }
};

}  // namespace

extern "C" const char *aspis_status_str(int status)
{
    switch (status) {
    case ASPIS_OK: return "ok";
    case ASPIS_E_INVAL: return "invalid argument";
    case ASPIS_E_RANGE: return "size out of supported range";
    case ASPIS_E_ALIGN: return "misaligned buffer";
    case ASPIS_E_CUDA: return "CUDA error";
    case ASPIS_E_LIMIT: return "clique search budget exhausted";
    case ASPIS_E_EMPTY: return "no file selected for aggregation";
    case ASPIS_E_NOT_IMPLEMENTED: return "not implemented";
    default: return "unknown status";
    }
}

extern "C" int aspis_abi_version(void) { return 2; }

// No call needs device workspace: the per-round intermediates are caller
// buffers and the kernels' working sets live in shared memory.
extern "C" size_t aspis_workspace_bytes(const aspis_assignment *) { return 0; }

extern "C" aspis_status aspis_assign(int K, int r, aspis_assignment *out)
{
    if (!out) return ASPIS_E_INVAL;
    std::memset(out, 0, sizeof(*out));
    if (r < 2 || K < r) return ASPIS_E_INVAL;
    if (K > ASPIS_MAX_K || r > ASPIS_MAX_R) return ASPIS_E_RANGE;
    const int64_t f = choose(K, r), l = choose(K - 1, r - 1);
    uint8_t *fw = (uint8_t *)std::malloc((size_t)(f * r));
    int32_t *wf = (int32_t *)std::malloc(sizeof(int32_t) * (size_t)(K * l));
    uint8_t *so = (uint8_t *)std::malloc((size_t)(K * l));
    if (!fw || !wf || !so) {
        std::free(fw);
        std::free(wf);
        std::free(so);
        return ASPIS_E_RANGE;
    }
    SubsetWriter gen{K, r, fw};
    gen.walk(0, 0);
    // invert the table: files of each worker in ascending file order
    std::vector<int64_t> fill((size_t)K, 0);
    for (int64_t i = 0; i < f; ++i)
        for (int s = 0; s < r; ++s) {
            const int j = fw[i * r + s];
            wf[(int64_t)j * l + fill[j]] = (int32_t)i;
            so[(int64_t)j * l + fill[j]] = (uint8_t)s;
            ++fill[j];
        }
    out->K = K;
    out->r = r;
    out->f = f;
    out->l = l;
    out->pair_share = choose(K - 2, r - 2);
    out->file_workers = fw;
    out->worker_files = wf;
    out->slot_of = so;
    out->dev_file_workers = nullptr;
    return ASPIS_OK;
}
